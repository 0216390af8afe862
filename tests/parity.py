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
    flagged sequences are counted and only checked for validity.
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


def compare_decision(res, gpu, inp_mask_before, cu_rows):
    """res: oracle StepResult; gpu: fetched dict."""
    B = len(cu_rows) - 1
    flagged = 0
    for b in range(B):
        r0, r1 = int(cu_rows[b]), int(cu_rows[b + 1])
        sl = slice(r0, r1)
        if res.flag_accept[b] or res.flag_lbs[b]:
            flagged += 1
            acc = gpu["accepted"][sl].astype(bool)
            assert np.all(inp_mask_before[sl][acc] == 1), "commit of an unmasked row"
            assert np.all(gpu["tokens"][sl][acc] == gpu["argmax"][sl][acc]), "commit value != x_hat"
            if inp_mask_before[sl].any() and (gpu["blk_meta"][b][1] > 0 or acc.any()):
                assert acc.sum() >= 1
            continue
        if not res.flag_lbs[b]:
            _close(f"lbs_logit[{b}]", gpu["lbs_logit"][sl], res.lbs_logit[sl])
        _close(f"lps_prob[{b}]", gpu["lps_prob"][sl], res.lps_prob[sl])
        for k in ("accepted", "tokens", "mask", "in_block"):
            g, o = np.asarray(gpu[k][sl]), np.asarray(getattr(res, k)[sl])
            assert np.array_equal(g.astype(np.int64), o.astype(np.int64)), \
                f"{k} differs in sequence {b}: gpu {g} oracle {o}"
        assert np.array_equal(gpu["blk_meta"][b], res.blk_meta[b]), \
            f"blk_meta differs in sequence {b}: {gpu['blk_meta'][b]} vs {res.blk_meta[b]}"
    return {"flagged_sequences": flagged, "sequences": B}
