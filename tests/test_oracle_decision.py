"""Pins of the oracle's EB decision (no GPU): hand-worked cases of the
filters and of the accept rule (tests/golden/*.json), the contiguity property
that Sec. 6.4 states for g_max = 1, structural properties of the block
selection over every small case, and the loop invariants of the App. E
algorithm (masked count never increases, at least one commit per step while
the block has masked rows, commits lie in B n M and take x_hat, termination
within L steps)."""
import itertools
import json
import os

import numpy as np
import pytest

import synth
from oracle import ebd_oracle as o

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _stats(conf, argmax, near=None):
    n = len(conf)
    conf = np.asarray(conf, float)
    return o.RowStats(conf=conf, entropy=np.zeros(n), ent_norm=np.zeros(n),
                      gap=np.zeros(n), argmax=np.asarray(argmax, np.int64),
                      logit_gap=np.ones(n), near_tie=np.zeros(n, bool)
                      if near is None else np.asarray(near, bool))


def test_maxgap_golden():
    g = json.load(open(os.path.join(GOLD, "block_selection.json")))
    for c in g["maxgap"]:
        assert o.max_gap_filter(c["C"], c["g_max"]) == c["B"], c


def test_select_golden():
    g = json.load(open(os.path.join(GOLD, "block_selection.json")))
    for c in g["select"]:
        prm = o.DecisionParams(tau=0.9, tau_psi=0.9, l_min=c["l_min"], l_b=c["l_b"],
                               g_max=c["g_max"], eos_id=c["eos"])
        M = [i for i, m in enumerate(c["mask"]) if m]
        O = np.array([c["O"][i] for i in M], float) if len(M) > c["l_min"] else None
        B = o.select_block(np.array(c["pos"]), M, O, np.array(c["argmax"]), prm)
        assert B == c["B"], c["note"]


def test_select_golden_through_decide_sequence():
    """Same cases through the full per-sequence step with an injected router."""
    g = json.load(open(os.path.join(GOLD, "block_selection.json")))
    for c in g["select"]:
        prm = o.DecisionParams(tau=2.0, tau_psi=2.0, l_min=c["l_min"], l_b=c["l_b"],
                               g_max=c["g_max"], eos_id=c["eos"], lps_enabled=False)
        n = len(c["pos"])
        mask = np.array(c["mask"], np.uint8)
        tokens = np.full(n, -1, np.int32)
        ib = np.zeros(n, np.uint8)
        meta = np.zeros(2, np.int32)
        Ofull = np.array(c["O"], float)
        d = o.decide_sequence(np.array(c["pos"]), mask, tokens, ib, meta,
                              _stats(np.linspace(0.1, 0.2, n), c["argmax"]), None, {},
                              prm, lbs_fn=lambda h, x: Ofull[np.array(c["mask"]) == 1])
        B = c["B"]
        want_meta = [0, 0] if len(B) == 1 else [c["pos"][B[0]], len(B)]
        assert meta.tolist() == want_meta, c["note"]
        # tau unreachable and LPS off: anti-stall commits the highest-kappa
        # row of B (kappa increases with the row index here)
        assert d.accepted.sum() == 1 and int(np.argmax(d.accepted)) == max(B)
        if len(B) > 1:
            assert np.flatnonzero(ib).tolist() == B


def test_accept_golden():
    g = json.load(open(os.path.join(GOLD, "accept.json")))
    for c in g["cases"]:
        prm = o.DecisionParams(tau=c["tau"], tau_psi=0.5, l_min=1, l_b=4, g_max=5,
                               eos_id=-7, lps_enabled=False)
        n = len(c["conf"])
        mask = np.array(c["mask"], np.uint8); tokens = np.full(n, -1, np.int32)
        ib = np.array(c["in_block"], np.uint8); meta = np.array(c["meta"], np.int32)
        d = o.decide_sequence(np.arange(n) + 50, mask, tokens, ib, meta,
                              _stats(c["conf"], c["argmax"]), None, {}, prm)
        assert d.accepted.tolist() == c["accepted"], c["note"]
        assert tokens.tolist() == c["tokens"], c["note"]
        assert mask.tolist() == c["mask_after"], c["note"]
        assert meta.tolist() == c["meta_after"], c["note"]


def _longest_valid_prefix(C, g):
    for k in range(len(C), -1, -1):
        if all(C[j + 1] - C[j] <= g for j in range(k - 1)):
            return C[:k]


def test_maxgap_exhaustive_and_contiguity():
    for n in range(0, 13):
        for bits in range(1 << n):
            C = [i for i in range(n) if bits >> i & 1]
            for g in (1, 2, 3, 5):
                B = o.max_gap_filter(C, g)
                assert B == _longest_valid_prefix(C, g)
                if g == 1 and B:
                    assert B == list(range(B[0], B[0] + len(B)))   # Sec. 6.4


def test_select_properties_exhaustive():
    """Over all masks and router sign patterns of 9 rows: B is a subset of M;
    |M| <= L_min gives B = M; otherwise |B| >= min(L_min, |M|) and either B is
    a gap-valid subset of the non-EOS router candidates starting at the first
    candidate, or the min-tokens fallback."""
    n, l_min, l_b, g = 9, 3, 5, 2
    prm = o.DecisionParams(tau=0.9, tau_psi=0.9, l_min=l_min, l_b=l_b, g_max=g, eos_id=7)
    pos = np.array([0, 1, 2, 4, 5, 9, 10, 11, 12])
    argmax = np.array([1, 7, 1, 1, 1, 1, 7, 1, 1])
    for mbits in range(1 << n):
        M = [i for i in range(n) if mbits >> i & 1]
        if len(M) <= l_min:
            assert o.select_block(pos, M, None, argmax, prm) == M
            continue
        for obits in range(1 << len(M)):
            O = np.array([1.0 if obits >> j & 1 else -1.0 for j in range(len(M))])
            B = o.select_block(pos, M, O, argmax, prm)
            assert set(B) <= set(M) and B == sorted(B)
            C = [i for j, i in enumerate(M) if O[j] > 0 and argmax[i] != 7]
            fallback = M[:min(l_b, len(M))]
            gaps_ok = all(pos[B[k + 1]] - pos[B[k]] <= g for k in range(len(B) - 1))
            stops = len(B) == len(C) or (0 < len(B) < len(C) and
                                         pos[C[len(B)]] - pos[B[-1]] > g)
            router_ok = (len(B) >= l_min and B == C[:len(B)] and gaps_ok and stops)
            assert router_ok or B == fallback
            if not router_ok:
                # the router branch must have produced fewer than L_min rows
                k = 1 if C else 0
                while k < len(C) and pos[C[k]] - pos[C[k - 1]] <= g:
                    k += 1
                assert k < l_min


def _random_seq(rng, n, lps=True):
    prm = o.DecisionParams(tau=0.9, tau_psi=0.6, l_min=4, l_b=8, g_max=3, eos_id=5,
                           lps_enabled=lps)
    pos = np.sort(rng.choice(200, n, replace=False)) + 1000
    mask = (rng.random(n) < 0.7).astype(np.uint8)
    return prm, pos, mask


def test_step_invariants_random():
    W = o.weights_f64(synth.router_weights(21, 32, 64))
    emb = synth.f32_to_bf16_bits(np.random.default_rng(22).standard_normal((16, 32)))
    rng = np.random.default_rng(23)
    for trial in range(60):
        n = int(rng.integers(1, 40))
        prm, pos, mask = _random_seq(rng, n, lps=bool(trial % 2))
        tokens = np.where(mask == 1, -1, rng.integers(0, 16, n)).astype(np.int32)
        ib = np.zeros(n, np.uint8); meta = np.zeros(2, np.int32)
        for stp in range(3 * n + 2):
            conf = rng.random(n) ** 3
            st = o.RowStats(conf=conf, entropy=-np.log(conf), ent_norm=rng.random(n),
                            gap=conf * rng.random(n), argmax=rng.integers(0, 16, n),
                            logit_gap=np.ones(n), near_tie=np.zeros(n, bool))
            m0, ib0 = mask.copy(), ib.copy()
            had_block = meta[1] > 0
            d = o.decide_sequence(pos, mask, tokens, ib, meta, st, emb, W, prm)
            acc = d.accepted.astype(bool)
            assert mask.sum() <= m0.sum()                         # never increases
            assert np.all(m0[acc] == 1)                            # commits were masked
            assert np.all(tokens[acc] == st.argmax[acc])          # commit value = x_hat
            assert np.all(mask[acc] == 0)
            if had_block:
                assert np.all(ib0[acc] == 1)                       # commits lie in B
                if np.any(m0[ib0 == 1] == 1):
                    assert acc.sum() >= 1                          # progress
            else:
                if ib.sum() > 0:
                    assert np.all(ib[acc] == 1)
                    assert np.all(ib <= m0)                        # new B within M
                if m0.sum() > 0:
                    assert acc.sum() >= 1
            if meta[1] == 0:
                assert ib.sum() == 0
            if mask.sum() == 0:
                break
        assert mask.sum() == 0, "loop did not terminate"


def test_small_generation_loop_terminates_within_L():
    sh = synth.tiny.with_(name="loop_tiny", prefix=16, gen_len=48, d_model=64,
                          vocab=512, n_heads_q=2, n_heads_kv=2, head_dim=16)
    W = o.weights_f64(synth.router_weights(sh.seed, sh.d_base, sh.gen_len))
    wl = synth.normal_bf16(1, 1, (sh.vocab, sh.d_model), 0.1)
    we = synth.normal_bf16(1, 2, (sh.vocab, sh.d_base), 1.0)
    prm = o.DecisionParams(tau=sh.tau, tau_psi=sh.tau_psi, l_min=sh.l_min, l_b=sh.l_b,
                           g_max=sh.g_max, eos_id=sh.eos_id)
    tokens, steps, commits, recs = o.generation_loop(
        sh, W, prm, lambda s, p: synth.loop_window_inputs(sh, s, p),
        lambda p: synth.loop_kv(sh, p), wl, we, attention=True)
    assert (tokens >= 0).all() and steps <= sh.gen_len
    assert all(c >= 1 for c in commits) and sum(commits) == sh.gen_len
    assert all(r["window"][1] - r["window"][0] <= 64 for r in recs)


def test_full_sequence_loop_invariants():
    """The full-sequence setting: every step's window is the whole response,
    M is every masked position.  The loop ends within L steps, commits at
    least one position per step, commits only masked positions of the
    window, and never unmasks anything else."""
    sh = synth.tiny.with_(name="loop_full", prefix=16, gen_len=80, d_model=64,
                          vocab=512, n_heads_q=2, n_heads_kv=2, head_dim=16, seed=3)
    W = o.weights_f64(synth.router_weights(sh.seed, sh.d_base, sh.gen_len))
    wl = synth.normal_bf16(3, 1, (sh.vocab, sh.d_model), 0.1)
    we = synth.normal_bf16(3, 2, (sh.vocab, sh.d_base), 1.0)
    prm = o.DecisionParams(tau=sh.tau, tau_psi=sh.tau_psi, l_min=sh.l_min, l_b=sh.l_b,
                           g_max=sh.g_max, eos_id=sh.eos_id)
    seen = []
    tokens, steps, commits, recs = o.generation_loop(
        sh, W, prm, lambda s, p: synth.loop_window_inputs(sh, s, p),
        lambda p: synth.loop_kv(sh, p), wl, we, window="full",
        on_step=lambda s, r: seen.append(r["accepted"].copy()))
    assert (tokens >= 0).all() and steps <= sh.gen_len
    assert all(c >= 1 for c in commits) and sum(commits) == sh.gen_len
    assert all(r["window"] == (0, sh.gen_len) for r in recs)
    committed = np.zeros(sh.gen_len, bool)
    for acc in seen:
        acc = acc.astype(bool)
        assert not np.any(committed & acc), "a position was committed twice"
        committed |= acc
    assert committed.all()
    assert any(r["lbs_ran"] for r in recs), "the LBS never ran on the whole response"


def _lps_feature_case(c):
    """Runs the per-sequence step on a golden case of lps_features.json with
    the LPS logit replaced by 0 (p_psi = 1/2, below tau_psi); returns the
    feature tuples the router received and the rows it scored."""
    n = len(c["pos"])
    seen = []

    def capture(feats):
        seen.append(np.array(feats, dtype=np.float64))
        return np.zeros(len(feats))
    st = o.RowStats(conf=np.array(c["conf"], float), entropy=np.zeros(n),
                    ent_norm=np.array(c["ent_norm"], float), gap=np.array(c["gap"], float),
                    argmax=np.arange(n, dtype=np.int64) + 100, logit_gap=np.ones(n),
                    near_tie=np.zeros(n, bool))
    prm = o.DecisionParams(tau=0.9, tau_psi=0.9, l_min=8, l_b=32, g_max=5, eos_id=-1)
    d = o.decide_sequence(np.array(c["pos"]), np.array(c["mask"], np.uint8),
                          np.full(n, -1, np.int32), np.array(c["in_block"], np.uint8),
                          np.array(c["meta"], np.int32), st, None, {}, prm, lps_fn=capture)
    assert len(seen) == 1
    return seen[0], np.flatnonzero(~np.isnan(d.lps_prob)).tolist()


def test_lps_feature_tuple_golden():
    """The LPS input tuple (kappa, H~, Delta, rho, pos) of every still-masked
    row of the block, in ascending position (Sec. 5.2, App. E; Readings R4,
    R5, R13), against hand-worked values."""
    g = json.load(open(os.path.join(GOLD, "lps_features.json")))
    for c in g["cases"]:
        feats, rows = _lps_feature_case(c)
        assert rows == c["rows"], c["note"]
        np.testing.assert_allclose(feats, np.array(c["features"]), rtol=0, atol=1e-15,
                                   err_msg=c["note"])
