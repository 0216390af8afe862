"""Comparison of the CUDA path with the CPU oracle.

Rules (spec parity bar):
  * conf, entropy, H~, Delta, attention output, router outputs: absolute
    difference <= 2e-3;
  * argmax: exact, except rows the oracle flags as near-ties (top-2 logit gap
    < 1e-3), where the GPU's choice must still be a logit within 1e-3 of the
    maximum;
  * accepted set, tokens, mask, block state: exact for every sequence the
    oracle does not flag (a near-tie on kappa vs tau, p_psi vs tau_psi,
    |O_phi|, the anti-stall argmax or an argmax feeding the decision);
    flagged sequences are counted; every sequence, flagged or not, must
    also be the decision that the rules give on the GPU's own router outputs
    and features (check_decision_valid).
"""
from __future__ import annotations

import numpy as np

TOL = 2e-3


def _close(name, a, b, tol=TOL, mask=None):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    if mask is not None:
        a, b = a[mask], b[mask]
    nan_a, nan_b = np.isnan(a), np.isnan(b)
    assert np.array_equal(nan_a, nan_b), f"{name}: NaN pattern differs"
    d = np.abs(a[~nan_a] - b[~nan_b])
    if d.size:
        i = int(np.argmax(d))
        assert d.max() <= tol, f"{name}: max |diff| {d.max():.3e} > {tol} at {i}"
    return float(d.max()) if d.size else 0.0


def compare_stats(st, gpu, rows=None, logits=None):
    """st: oracle RowStats for the compared rows; gpu: dict of arrays over the
    same rows."""
    rep = {}
    rep["conf"] = _close("conf", gpu["conf"], st.conf)
    rep["entropy"] = _close("entropy", gpu["entropy"], st.entropy)
    rep["ent_norm"] = _close("ent_norm", gpu["ent_norm"], st.ent_norm)
    rep["gap"] = _close("gap", gpu["gap"], st.gap)
    nt = np.asarray(st.near_tie, bool)
    am = np.asarray(gpu["argmax"], np.int64)
    bad = (am != st.argmax) & ~nt
    assert not bad.any(), f"argmax differs at rows {np.flatnonzero(bad)[:8]}"
    if logits is not None and nt.any():
        for r in np.flatnonzero(nt):
            assert logits[r].max() - logits[r][am[r]] < 1e-3, "near-tie argmax off the top set"
    rep["argmax_near_ties"] = int(nt.sum())
    return rep


def check_decision_valid(pos, m0, t0, ib0, meta0, g, meta_out, prm):
    """The GPU's decision for one sequence, re-derived from the GPU's own
    router outputs and features with the rules of the App. E algorithm, must
    match exactly.  pos/m0/t0/ib0/meta0: the sequence's positions and
    decode state before the step; g: the GPU's per-row outputs of the step
    (conf, argmax, lbs_logit, lps_prob, accepted, tokens, mask, in_block)
    over the sequence's rows; meta_out: the GPU's block state after it; prm:
    oracle DecisionParams.  Needs no oracle statistics, so it holds for
    sequences flagged for a near-tie too.  Checked:
      * commits are masked rows of the step's block B, take x_hat, and no
        other row's token or mask changes;
      * with no active block, B is what the filters (size fallback, EOS
        removal, MaxGapFilter, min-tokens fallback) give on the GPU's router
        logits and argmax; with one, B is the active block and the LBS did
        not run;
      * the accepted set is the union rule (kappa >= tau or p_psi > tau_psi,
        compared in float32 as the GPU compares) on B n M, or the anti-stall
        row (highest kappa, lowest position on ties);
      * the block state after the step: B with b = min B and |B| frozen at
        selection while B keeps masked rows, cleared otherwise."""
    from oracle import ebd_oracle as o
    n = len(pos)
    m0 = np.asarray(m0).astype(bool)
    acc = np.asarray(g["accepted"]).astype(bool)
    am = np.asarray(g["argmax"], np.int64)
    assert np.all(m0[acc]), "commit of an unmasked row"
    assert np.array_equal(np.asarray(g["tokens"])[acc], am[acc]), "commit value != x_hat"
    assert not np.asarray(g["mask"])[acc].any(), "committed row still masked"
    assert np.array_equal(np.asarray(g["tokens"])[~acc], np.asarray(t0)[~acc]), "uncommitted token changed"
    assert np.array_equal(np.asarray(g["mask"])[~acc].astype(bool), m0[~acc]), "uncommitted mask changed"
    M = [i for i in range(n) if m0[i]]
    O = np.asarray(g["lbs_logit"], np.float64)
    if meta0[1] > 0:                                   # active block
        B = [i for i in range(n) if ib0[i]]
        assert np.all(np.isnan(O)), "the LBS ran inside an active block"
        b_meta = (int(meta0[0]), int(meta0[1]))
    else:                                              # block selection
        ran = len(M) > prm.l_min
        assert np.array_equal(np.isfinite(O), np.isin(np.arange(n), M) & ran), "LBS rows"
        B = o.select_block(np.asarray(pos), M, O[M] if ran else None, am, prm)
        b_meta = (int(pos[B[0]]), len(B)) if B else (0, 0)
    BM = [i for i in B if m0[i]]
    conf = np.asarray(g["conf"], np.float32)
    lps = np.asarray(g["lps_prob"], np.float32)
    if BM:
        A = [i for i in BM if conf[i] >= np.float32(prm.tau) or
             (prm.lps_enabled and lps[i] > np.float32(prm.tau_psi))]
        if not A:
            A = [max(BM, key=lambda i: (conf[i], -i))]
    else:
        A = []
    assert sorted(np.flatnonzero(acc).tolist()) == sorted(A), f"accepted {np.flatnonzero(acc)} vs rules {A}"
    still = [i for i in B if m0[i] and not acc[i]]
    ib_out = np.asarray(g["in_block"]).astype(bool)
    if still:
        assert np.array_equal(ib_out, np.isin(np.arange(n), B)), "block rows after the step"
        assert (int(meta_out[0]), int(meta_out[1])) == b_meta, f"blk_meta {meta_out} vs {b_meta}"
    else:
        assert not ib_out.any() and tuple(int(x) for x in meta_out) == (0, 0), "resolved block not cleared"


def compare_decision(res, gpu, inp, prm):
    """res: oracle StepResult; gpu: fetched dict; inp: the step's inputs
    (decode state before the step); prm: oracle DecisionParams.  Every
    sequence passes check_decision_valid; the ones the oracle does not flag
    must also equal the oracle exactly."""
    cu_rows = inp.cu_rows
    B = len(cu_rows) - 1
    flagged = 0
    for b in range(B):
        r0, r1 = int(cu_rows[b]), int(cu_rows[b + 1])
        sl = slice(r0, r1)
        g = {k: gpu[k][sl] for k in ("conf", "argmax", "lbs_logit", "lps_prob", "accepted",
                                      "tokens", "mask", "in_block")}
        if not np.all(np.asarray(gpu["argmax"][sl]) >= 0):
            continue  # a non-finite row (EBD_ERR_NONFINITE): checked by its own test
        check_decision_valid(inp.row_pos[sl], inp.mask[sl], inp.tokens[sl], inp.in_block[sl],
                             inp.blk_meta[b], g, gpu["blk_meta"][b], prm)
        if res.flag_accept[b] or res.flag_lbs[b]:
            flagged += 1
            continue
        _close(f"lbs_logit[{b}]", gpu["lbs_logit"][sl], res.lbs_logit[sl])
        _close(f"lps_prob[{b}]", gpu["lps_prob"][sl], res.lps_prob[sl])
        for k in ("accepted", "tokens", "mask", "in_block"):
            gg, oo = np.asarray(gpu[k][sl]), np.asarray(getattr(res, k)[sl])
            assert np.array_equal(gg.astype(np.int64), oo.astype(np.int64)), \
                f"{k} differs in sequence {b}: gpu {gg} oracle {oo}"
        assert np.array_equal(gpu["blk_meta"][b], res.blk_meta[b]), \
            f"blk_meta differs in sequence {b}: {gpu['blk_meta'][b]} vs {res.blk_meta[b]}"
    return {"flagged_sequences": flagged, "sequences": B}
