"""The full-sequence setting on the GPU through the C ABI: every position of
the response is a row of the step and the LBS sees every masked position
(App. E algorithm with M = all masked positions; windows of up to 512 rows
per sequence, decided by the grid-wide decision kernels).

* tiny shape, 3 sequences of 256, 100 and 40 rows: the whole step against
  the oracle (statistics of every row; routers, block, commit exact unless
  flagged for a near-tie), with no active block and inside a block, and the
  baselines' rules;
* LLaDA-8B shape, one 512-row response: statistics on sampled rows and the
  decision against the oracle's on the GPU's statistics;
* the tiny full-sequence generation loop step by step against the oracle's;
* a window of at most 64 rows decided by both decision paths gives the same
  decision."""
import numpy as np
import pytest

import synth
from oracle import ebd_oracle as o
from tests import parity

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

MODES = {"eb": 0, "threshold": 1, "topm": 2}


def _prm(sh):
    return o.DecisionParams(tau=sh.tau, tau_psi=sh.tau_psi, l_min=sh.l_min, l_b=sh.l_b,
                            g_max=sh.g_max, eos_id=sh.eos_id, lps_enabled=bool(sh.lps_enabled))


def _gpu_step(sh, inp, max_window=None, mode="eb", top_m=1):
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    w = rt.upload_weights(inp)
    cfg = rt.config_for(sh, max_window=max_window, decode_mode=MODES[mode], top_m=top_m)
    h = rt.Handle(cfg, w.w_emb)
    try:
        ds = rt.DeviceStep(inp, w, attention=False)
        E.check(E.ebd_step(h.h, ds.args(), rt.stream_handle(None)), h.h)
        assert h.sync_status() == 0, E.ebd_last_error(h.h)
        return ds.fetch()
    finally:
        h.close()


def _injected(inp, gpu, sh):
    R = inp.rows
    return o.RowStats(conf=gpu["conf"].astype(np.float64), entropy=gpu["entropy"].astype(np.float64),
                      ent_norm=gpu["ent_norm"].astype(np.float64), gap=gpu["gap"].astype(np.float64),
                      argmax=gpu["argmax"].astype(np.int64), logit_gap=np.full(R, np.inf),
                      near_tie=np.zeros(R, bool))


def _weights(sh):
    return o.weights_f64(synth.router_weights(sh.seed, sh.d_base, sh.gen_len))


@pytest.mark.parametrize("state", ["select", "inblock"])
def test_tiny_full_step_matches_oracle(state):
    sh = synth.tiny_full
    inp = synth.make_step_inputs(sh)
    if state == "inblock":
        synth.preset_in_block(inp, 24)
    gpu = _gpu_step(sh, inp)
    res = o.step(inp, _weights(sh), _prm(sh), attention=False)
    parity.compare_stats(res.stats, gpu)
    rep = parity.compare_decision(res, gpu, inp, _prm(sh))
    assert rep["flagged_sequences"] < rep["sequences"]
    if state == "select":
        assert np.any(np.isfinite(gpu["lbs_logit"])), "the LBS did not run"
    assert np.any(np.isfinite(gpu["lps_prob"])), "the LPS did not run"


@pytest.mark.parametrize("mode,top_m", [("threshold", 1), ("topm", 7)])
def test_tiny_full_baselines(mode, top_m):
    sh = synth.tiny_full
    inp = synth.make_step_inputs(sh)
    gpu = _gpu_step(sh, inp, mode=mode, top_m=top_m)
    st = _injected(inp, gpu, sh)
    for b in range(len(inp.cu_rows) - 1):
        r0, r1 = int(inp.cu_rows[b]), int(inp.cu_rows[b + 1])
        m, t = inp.mask[r0:r1].copy(), inp.tokens[r0:r1].copy()
        sub = o.RowStats(*(getattr(st, f)[r0:r1] for f in
                           ("conf", "entropy", "ent_norm", "gap", "argmax", "logit_gap", "near_tie")))
        d = o.decide_fixed_block(m, t, sub, mode, sh.tau, top_m)
        if d.flag_accept:
            continue
        assert np.array_equal(gpu["accepted"][r0:r1], d.accepted), b
        assert np.array_equal(gpu["mask"][r0:r1], m) and np.array_equal(gpu["tokens"][r0:r1], t), b
    assert np.all(np.isnan(gpu["lbs_logit"])) and np.all(np.isnan(gpu["lps_prob"]))
    assert np.array_equal(gpu["in_block"], inp.in_block) and np.array_equal(gpu["blk_meta"], inp.blk_meta)


def test_llada_full_step_512_rows():
    sh = synth.llada_full
    inp = synth.make_step_inputs(sh)
    gpu = _gpu_step(sh, inp)
    rows = np.array([0, 1, 255, 256, 510, 511])
    st = o.softmax_stats(o.lm_logits(inp.hidden[rows], inp.w_lm))
    parity.compare_stats(st, {k: gpu[k][rows] for k in ("conf", "entropy", "ent_norm", "gap", "argmax")})
    res = o.decide(inp.cu_rows, inp.row_pos, inp.tokens, inp.mask, inp.in_block, inp.blk_meta,
                   _injected(inp, gpu, sh), inp.w_emb, _weights(sh), _prm(sh))
    parity.compare_decision(res, gpu, inp, _prm(sh))
    assert np.isfinite(gpu["lbs_logit"][inp.mask == 1]).all()


def test_full_loop_tiny_matches_oracle():
    from paper_2609_16450_gb300 import loop as lp
    from paper_2609_16450_gb300 import runtime as rt
    sh = synth.loop_full_tiny
    inp = synth.make_step_inputs(sh)
    w = rt.upload_weights(inp)
    h = rt.Handle(lp.config_for_loop(sh, max_window=sh.gen_len), w.w_emb)
    try:
        res = lp.run_loop(h, sh, w, lambda s, p: synth.loop_window_inputs(sh, s, p),
                          lambda p: synth.loop_kv(sh, p), attention=False, window="full")
    finally:
        h.close()
    toks, steps, commits, recs = o.generation_loop(
        sh, _weights(sh), _prm(sh), lambda s, p: synth.loop_window_inputs(sh, s, p),
        lambda p: synth.loop_kv(sh, p), inp.w_lm, inp.w_emb, window="full")
    assert sum(res.commits) == sh.gen_len and all(c >= 1 for c in res.commits)
    compared = 0
    for g, r in zip(res.records, recs):
        assert g.window == r["window"] == (0, sh.gen_len)
        st = r["stats"]
        for k in ("conf", "entropy", "gap"):
            parity._close(f"{k} step {g.step}", getattr(g, k), getattr(st, k))
        if r["flag"] or r["flag_lbs"]:
            break
        assert np.array_equal(g.accepted, r["accepted"]), g.step
        compared += 1
    else:
        assert res.steps == steps and np.array_equal(res.tokens, toks)
    assert compared >= 1


def test_small_window_same_decision_on_both_paths():
    """The LLaDA-8B-shaped selection step (32 rows) decided by the cluster
    kernel (max_window 64) and by the grid-wide kernels (max_window 128)."""
    sh = synth.llada
    inp = synth.make_step_inputs(sh)
    a = _gpu_step(sh, inp)
    b = _gpu_step(sh, inp, max_window=128)
    for k in ("accepted", "tokens", "mask", "in_block", "blk_meta", "argmax"):
        assert np.array_equal(a[k], b[k]), k
    for k in ("conf", "entropy", "gap", "lbs_logit", "lps_prob"):
        parity._close(k, a[k], b[k])
