"""Pins of the oracle's fixed-block rules of the baselines (App. B,
Eq. prelim-update): hand-worked cases (tests/golden/baseline_rules.json),
the defining properties of Top-m and of the threshold rule on random
blocks, and loop invariants (Top-1 takes exactly one step per position;
the threshold rule never takes more steps than Top-1)."""
import json
import os

import numpy as np

import synth
from oracle import ebd_oracle as o

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _stats(conf, argmax):
    n = len(conf)
    return o.RowStats(conf=np.asarray(conf, float), entropy=np.zeros(n), ent_norm=np.zeros(n),
                      gap=np.zeros(n), argmax=np.asarray(argmax, np.int64),
                      logit_gap=np.ones(n), near_tie=np.zeros(n, bool))


def test_golden_cases():
    g = json.load(open(os.path.join(GOLD, "baseline_rules.json")))
    for c in g["cases"]:
        n = len(c["conf"])
        mask = np.array(c["mask"], np.uint8)
        tokens = np.full(n, -1, np.int32)
        d = o.decide_fixed_block(mask, tokens, _stats(c["conf"], c["argmax"]), c["mode"],
                                 c["tau"], c["m"])
        assert d.accepted.tolist() == c["accepted"], c["note"]
        assert tokens.tolist() == c["tokens"], c["note"]
        assert np.all(mask[np.array(c["accepted"], bool)] == 0)


def test_golden_windows():
    g = json.load(open(os.path.join(GOLD, "baseline_rules.json")))
    for c in g["windows"]:
        assert list(o.fixed_block_window(np.array(c["mask"]), c["block"])) == c["window"], c


def test_rule_properties_on_random_blocks():
    rng = np.random.default_rng(3)
    for _ in range(500):
        n = int(rng.integers(1, 40))
        conf = np.round(rng.random(n), 2)  # coarse values: ties occur
        mask = (rng.random(n) < 0.7).astype(np.uint8)
        M = np.flatnonzero(mask)
        st = _stats(conf, rng.integers(0, 100, n))
        m = int(rng.integers(1, 8))
        mk = mask.copy(); tk = np.full(n, -1, np.int32)
        A = np.flatnonzero(o.decide_fixed_block(mk, tk, st, "topm", 0.9, m).accepted)
        assert A.size == min(m, M.size)
        rest = np.setdiff1d(M, A)
        if A.size and rest.size:
            assert conf[A].min() >= conf[rest].max()
            # among equal kappa at the boundary the lower positions go first
            edge = conf[A].min()
            assert not np.any((conf[rest] == edge) & (rest < A[conf[A] == edge].max()))
        mk = mask.copy(); tk = np.full(n, -1, np.int32)
        A = np.flatnonzero(o.decide_fixed_block(mk, tk, st, "threshold", 0.9, 1).accepted)
        above = M[conf[M] >= 0.9]
        if above.size:
            assert np.array_equal(A, above)
        elif M.size:
            assert A.size == 1 and conf[A[0]] == conf[M].max()
            assert A[0] == M[conf[M] == conf[M].max()].min()
        assert np.all(mk[A] == 0) and np.all(tk[A] == st.argmax[A])


def test_loop_step_counts():
    sh = synth.loop_tiny.with_(gen_len=24, prefix=8)
    inp = synth.make_step_inputs(sh)
    W = o.weights_f64(synth.router_weights(sh.seed, sh.d_base, sh.gen_len))
    prm = o.DecisionParams(tau=sh.tau, tau_psi=sh.tau_psi, l_min=sh.l_min, l_b=sh.l_b,
                           g_max=sh.g_max, eos_id=sh.eos_id)
    win = lambda s, p: synth.loop_window_inputs(sh, s, p)
    kv = lambda p: synth.loop_kv(sh, p)
    runs = {}
    for mode, m in (("topm", 1), ("topm", 3), ("threshold", 1)):
        toks, steps, commits, recs = o.generation_loop(sh, W, prm, win, kv, inp.w_lm, inp.w_emb,
                                                       mode=mode, block=8, top_m=m)
        assert np.all(toks >= 0)
        assert sum(commits) == sh.gen_len and all(c >= 1 for c in commits)
        for r in recs:  # every window is one fixed block
            lo, hi = r["window"]
            assert lo % 8 == 0 and hi - lo <= 8
        runs[(mode, m)] = steps
    assert runs[("topm", 1)] == sh.gen_len
    assert runs[("topm", 3)] == sum(-(-8 // 3) for _ in range(sh.gen_len // 8))
    assert runs[("threshold", 1)] <= runs[("topm", 1)]
