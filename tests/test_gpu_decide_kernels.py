"""Both per-sequence decision kernels for windows of up to 32 rows -- one
8-CTA cluster per sequence, and one CTA per sequence with the LBS products
on tcgen05 -- against the oracle through the C ABI, each forced in turn with
EBD_DECIDE_KERNEL (without it, the launch's batch size picks the kernel).

* the tiny and LLaDA-8B steps with no active block (the LBS runs) and inside
  one; at LLaDA-8B with one sequence the LM head leaves SMs free, so the
  one-CTA kernel also runs its stand-in warm-up before the real window;
* one batch of degenerate windows (empty, one row, a full 32-row window, no
  cached prefix, nothing masked, |M| <= L_min) with and without a block;
* non-finite hidden rows (reported, not committed; other sequences exact);
* the router branches forced both ways by the head biases, EOS removal;
* the baselines' threshold and Top-m rules;
* sweep points of 16 and 64 sequences, where the batch rule picks the
  one-CTA kernel;
* ebd_decide (statistics as inputs) on a step's own statistics takes that
  step's decision bit for bit."""
import numpy as np
import pytest

import synth
from oracle import ebd_oracle as o
from tests import parity
from tests import test_gpu_baselines as B
from tests import test_gpu_configs as C
from tests import test_gpu_edges as G
from tests import test_gpu_step as S

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(params=["cta", "cluster"])
def kernel(request, monkeypatch):
    monkeypatch.setenv("EBD_DECIDE_KERNEL", request.param)
    return request.param


@pytest.mark.parametrize("state", ["select", "inblock"])
def test_tiny_step(kernel, state):
    S.test_tiny_step(state)


def test_llada_step(kernel):
    S.test_llada_step("packed")


def _ragged32(state):
    sh = synth.tiny.with_(name="edge32", batch=6, windows=(0, 1, 32, 7, 20, 24), seed=19)
    inp = synth.make_step_inputs(sh, prefix_lens=np.array([128, 0, 128, 5, 64, 128]))
    cu = inp.cu_rows
    r0, r1 = int(cu[4]), int(cu[5])  # nothing left to unmask
    inp.mask[r0:r1] = 0
    inp.tokens[r0:r1] = 7 + np.arange(r1 - r0)
    r0, r1 = int(cu[5]), int(cu[6])  # |M| = 5 <= L_min
    m = np.zeros(r1 - r0, np.uint8)
    m[[1, 4, 9, 10, 17]] = 1
    inp.mask[r0:r1] = m
    inp.tokens[r0:r1] = np.where(m == 1, -1, 11)
    assert sh.l_min >= int(m.sum())
    r0, r1 = int(cu[2]), int(cu[3])  # a full window, every row masked
    inp.mask[r0:r1] = 1
    inp.tokens[r0:r1] = -1
    if state == "inblock":
        synth.preset_in_block(inp, 16)
    return sh, inp


@pytest.mark.parametrize("state", ["select", "inblock"])
def test_degenerate_windows(kernel, state):
    sh, inp = _ragged32(state)
    gpu = G._step(sh, inp, max_window=32)
    res = o.step(inp, G._weights(sh), G._prm(sh))
    parity.compare_stats(res.stats, gpu)
    parity._close("attn_out", gpu["attn_out"], res.attn_out)
    rep = parity.compare_decision(res, gpu, inp, G._prm(sh))
    assert rep["flagged_sequences"] <= 2, rep
    cu = inp.cu_rows
    sl = slice(int(cu[4]), int(cu[5]))
    assert not gpu["accepted"][sl].any() and np.array_equal(gpu["tokens"][sl], inp.tokens[sl])
    assert tuple(gpu["blk_meta"][4]) == (0, 0)
    if state == "select":
        sl = slice(int(cu[5]), int(cu[6]))
        assert np.all(np.isnan(gpu["lbs_logit"][sl]))
        # the full window ran the LBS over all 32 rows
        sl = slice(int(cu[2]), int(cu[3]))
        assert np.all(np.isfinite(gpu["lbs_logit"][sl]))


def test_nonfinite_rows(kernel):
    G.test_nonfinite_rows_are_reported_and_not_committed(32)


@pytest.mark.parametrize("lbs_head,lps_head", [(4.0, 4.0), (-4.0, -4.0), (4.0, -4.0)])
def test_router_branches(kernel, lbs_head, lps_head):
    S.test_router_branches(lbs_head, lps_head)


def test_eos_removal(kernel):
    S.test_eos_removal()


@pytest.mark.parametrize("mode,top_m", [("threshold", 1), ("topm", 5)])
def test_baseline_modes(kernel, mode, top_m):
    B.test_llada_step_modes(mode, top_m)


@pytest.mark.parametrize("point", [(16, 256, 32), (64, 256, 8)])
def test_many_sequences(kernel, point):
    C.test_sweep_point(point)


@pytest.mark.parametrize("state", ["select", "inblock"])
def test_decide_entry_takes_the_steps_decision(kernel, state):
    """ebd_decide (statistics as inputs) on the statistics a step produced, from
    the same decode state, takes exactly that step's decision."""
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    sh = synth.llada
    inp = synth.make_step_inputs(sh)
    if state == "inblock":
        synth.preset_in_block(inp, 20)
    w = rt.upload_weights(inp)
    h = rt.Handle(rt.config_for(sh), w.w_emb)
    try:
        ds = rt.DeviceStep(inp, w, attention=False)
        E.check(E.ebd_step(h.h, ds.args(), rt.stream_handle(None)), h.h)
        assert h.sync_status() == 0
        step = ds.fetch()
        ds.restore_state()
        E.check(E.ebd_decide(h.h, ds.args(), rt.stream_handle(None)), h.h)
        assert h.sync_status() == 0
        dec = ds.fetch()
        for k in ("tokens", "mask", "in_block", "blk_meta", "accepted"):
            np.testing.assert_array_equal(dec[k], step[k], err_msg=k)
        for k in ("lbs_logit", "lps_prob"):
            np.testing.assert_array_equal(dec[k], step[k], err_msg=k)  # NaN where not scored
        assert step["accepted"].sum() >= 1
    finally:
        h.close()
