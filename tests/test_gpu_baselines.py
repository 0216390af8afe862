"""The baselines' fixed-block rules (App. B, Eq. prelim-update) as decode
modes of the decision kernel, against the oracle: the tiny generation loop
step by step under the threshold rule and under Top-m, and one LLaDA-8B
shaped step in each mode with the GPU's statistics fed to the oracle's
rule.  Also the step counts of the three decoders on the tiny loop."""
import numpy as np
import pytest

import synth
from oracle import ebd_oracle as o
from tests import parity

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

MODES = {"threshold": 1, "topm": 2}


def _prm(sh):
    return o.DecisionParams(tau=sh.tau, tau_psi=sh.tau_psi, l_min=sh.l_min, l_b=sh.l_b,
                            g_max=sh.g_max, eos_id=sh.eos_id, lps_enabled=bool(sh.lps_enabled))


def _gpu_loop(sh, inp, mode, top_m, block):
    from paper_2609_16450_gb300 import loop as lp
    from paper_2609_16450_gb300 import runtime as rt
    w = rt.upload_weights(inp)
    h = rt.Handle(lp.config_for_loop(sh, decode_mode=MODES.get(mode, 0), top_m=top_m), w.w_emb)
    try:
        return lp.run_loop(h, sh, w, lambda s, p: synth.loop_window_inputs(sh, s, p),
                           lambda p: synth.loop_kv(sh, p), attention=True, block=block)
    finally:
        h.close()


@pytest.mark.parametrize("mode,top_m", [("threshold", 1), ("topm", 1), ("topm", 4)])
def test_tiny_loop_matches_oracle(mode, top_m):
    sh = synth.loop_tiny
    inp = synth.make_step_inputs(sh)
    res = _gpu_loop(sh, inp, mode, top_m, 16)
    W = o.weights_f64(synth.router_weights(sh.seed, sh.d_base, sh.gen_len))
    toks, steps, commits, recs = o.generation_loop(
        sh, W, _prm(sh), lambda s, p: synth.loop_window_inputs(sh, s, p),
        lambda p: synth.loop_kv(sh, p), inp.w_lm, inp.w_emb, attention=True, mode=mode,
        block=16, top_m=top_m)
    assert sum(res.commits) == sh.gen_len
    for g, r in zip(res.records, recs):
        assert g.window == r["window"], (g.step, g.window, r["window"])
        parity._close(f"attn step {g.step}", g.attn_out, r["attn"])
        if r["flag"]:
            break
        assert np.array_equal(g.accepted, r["accepted"]), (g.step, g.accepted, r["accepted"])
        assert np.all(np.isnan(g.lbs_logit)) and np.all(np.isnan(g.lps_prob))
    else:
        assert res.steps == steps
        assert np.array_equal(res.tokens, toks)
    if mode == "topm":
        assert res.steps == sum(-(-16 // top_m) for _ in range(sh.gen_len // 16))


@pytest.mark.parametrize("mode,top_m", [("threshold", 1), ("topm", 5)])
def test_llada_step_modes(mode, top_m):
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    sh = synth.llada
    inp = synth.make_step_inputs(sh)
    w = rt.upload_weights(inp)
    h = rt.Handle(rt.config_for(sh, decode_mode=MODES[mode], top_m=top_m), w.w_emb)
    try:
        ds = rt.DeviceStep(inp, w)
        E.check(E.ebd_step(h.h, ds.args(), rt.stream_handle(None)), h.h)
        assert h.sync_status() == 0
        gpu = ds.fetch()
    finally:
        h.close()
    R = inp.rows
    st = o.RowStats(conf=gpu["conf"].astype(np.float64), entropy=gpu["entropy"].astype(np.float64),
                    ent_norm=gpu["ent_norm"].astype(np.float64), gap=gpu["gap"].astype(np.float64),
                    argmax=gpu["argmax"].astype(np.int64), logit_gap=np.full(R, np.inf),
                    near_tie=np.zeros(R, bool))
    mask, tokens = inp.mask.copy(), inp.tokens.copy()
    d = o.decide_fixed_block(mask, tokens, st, mode, sh.tau, top_m)
    if not d.flag_accept:
        assert np.array_equal(gpu["accepted"], d.accepted)
        assert np.array_equal(gpu["mask"], mask) and np.array_equal(gpu["tokens"], tokens)
    assert np.array_equal(gpu["in_block"], inp.in_block)
    assert np.array_equal(gpu["blk_meta"], inp.blk_meta)
    if mode == "topm":
        assert gpu["accepted"].sum() == min(top_m, int(inp.mask.sum()))


def test_step_counts_of_the_three_decoders():
    sh = synth.loop_tiny
    inp = synth.make_step_inputs(sh)
    steps = {m: _gpu_loop(sh, inp, m, 1, 32).steps for m in ("eb", "threshold", "topm")}
    print("tiny loop steps:", steps)
    assert steps["topm"] == sh.gen_len
    assert steps["threshold"] <= steps["topm"] and steps["eb"] <= steps["topm"]
