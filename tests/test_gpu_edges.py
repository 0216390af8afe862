"""Degenerate and ragged steps on the GPU through the C ABI, against the oracle.

* One batch that holds every degenerate sequence the step can see: an empty
  window (0 rows), a one-row window, a full 64-row window, a window with no
  cached prefix, a window with no masked row left, and one whose masked set
  is no larger than L_min (B = M without the LBS, Sec. 4.1).  The whole step
  (attention, statistics, routers, block, commit) against the oracle, with
  no active block and inside one, decided by the cluster kernel and by the
  grid-wide kernels.
* An empty step (rows = 0) returns EBD_OK and touches nothing.
* A hidden state with NaN or Inf: the step reports EBD_ERR_NONFINITE, the
  row's argmax is -1 and it stays masked, and every other sequence's
  decision is the oracle's."""
import numpy as np
import pytest

import synth
from oracle import ebd_oracle as o
from tests import parity

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

BF16_NAN, BF16_INF = 0x7FC0, 0x7F80


def _prm(sh):
    return o.DecisionParams(tau=sh.tau, tau_psi=sh.tau_psi, l_min=sh.l_min, l_b=sh.l_b,
                            g_max=sh.g_max, eos_id=sh.eos_id, lps_enabled=bool(sh.lps_enabled))


def _weights(sh):
    return o.weights_f64(synth.router_weights(sh.seed, sh.d_base, sh.gen_len))


def _ragged(state):
    sh = synth.tiny.with_(name="edge", batch=6, windows=(0, 1, 64, 7, 33, 20), seed=9)
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
    if state == "inblock":
        synth.preset_in_block(inp, 16)
    return sh, inp


def _step(sh, inp, max_window=None, attention=True, expect=0):
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    w = rt.upload_weights(inp)
    h = rt.Handle(rt.config_for(sh, max_window=max_window), w.w_emb)
    try:
        ds = rt.DeviceStep(inp, w, attention=attention)
        E.check(E.ebd_step(h.h, ds.args(), rt.stream_handle(None)), h.h)
        assert h.sync_status() == expect, E.ebd_last_error(h.h)
        return ds.fetch()
    finally:
        h.close()


@pytest.mark.parametrize("state", ["select", "inblock"])
@pytest.mark.parametrize("max_window", [64, 128])
def test_degenerate_sequences_match_oracle(state, max_window):
    sh, inp = _ragged(state)
    attention = max_window <= 64  # the grid-wide setting has no window attention
    gpu = _step(sh, inp, max_window=max_window, attention=attention)
    res = o.step(inp, _weights(sh), _prm(sh), attention=attention)
    parity.compare_stats(res.stats, gpu)
    if attention:
        parity._close("attn_out", gpu["attn_out"], res.attn_out)
    rep = parity.compare_decision(res, gpu, inp, _prm(sh))
    assert rep["flagged_sequences"] <= 2, rep
    cu = inp.cu_rows
    # nothing masked: no commit, no block
    sl = slice(int(cu[4]), int(cu[5]))
    assert not gpu["accepted"][sl].any() and np.array_equal(gpu["tokens"][sl], inp.tokens[sl])
    assert tuple(gpu["blk_meta"][4]) == (0, 0)
    if state == "select":
        # |M| <= L_min: the LBS does not run and the block is M
        sl = slice(int(cu[5]), int(cu[6]))
        assert np.all(np.isnan(gpu["lbs_logit"][sl]))
        if not (res.flag_accept[5] or res.flag_lbs[5]):
            assert gpu["blk_meta"][5][1] == 5 or gpu["blk_meta"][5][1] == 0


def test_empty_step_touches_nothing():
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    sh = synth.tiny
    inp = synth.make_step_inputs(sh)
    w = rt.upload_weights(inp)
    h = rt.Handle(rt.config_for(sh), w.w_emb)
    try:
        ds = rt.DeviceStep(inp, w)
        a = ds.args()
        before = ds.fetch()
        a.rows = 0
        E.check(E.ebd_step(h.h, a, rt.stream_handle(None)), h.h)
        a.batch = 0
        E.check(E.ebd_step(h.h, a, rt.stream_handle(None)), h.h)
        torch.cuda.synchronize()
        assert h.sync_status() == 0
        after = ds.fetch()
        for k, v in before.items():
            assert np.array_equal(np.asarray(v), np.asarray(after[k]), equal_nan=True), k
    finally:
        h.close()


@pytest.mark.parametrize("max_window", [64, 128])
def test_nonfinite_rows_are_reported_and_not_committed(max_window):
    from paper_2609_16450_gb300 import _ebd as E
    sh = synth.tiny.with_(name="nonfinite", batch=3, windows=(20, 32, 12), seed=5)
    inp = synth.make_step_inputs(sh)
    cu = inp.cu_rows
    bad_seq = 1
    bad = [int(cu[bad_seq]) + 2, int(cu[bad_seq]) + 5]
    clean = inp.hidden.copy()
    inp.hidden[bad[0]] = BF16_NAN
    inp.hidden[bad[1]] = BF16_INF
    attention = max_window <= 64
    gpu = _step(sh, inp, max_window=max_window, attention=attention, expect=E.EBD_ERR_NONFINITE)
    assert np.all(gpu["argmax"][bad] == -1)
    assert np.all(gpu["mask"][bad] == 1) and not gpu["accepted"][bad].any()
    assert np.array_equal(gpu["tokens"][bad], inp.tokens[bad])
    # every other sequence is decided as if the bad rows were not there
    inp.hidden = clean
    res = o.step(inp, _weights(sh), _prm(sh), attention=False)
    ok = np.ones(inp.rows, bool)
    ok[int(cu[bad_seq]):int(cu[bad_seq + 1])] = False
    sub = o.RowStats(*(np.asarray(getattr(res.stats, f))[ok] for f in
                       ("conf", "entropy", "ent_norm", "gap", "argmax", "logit_gap", "near_tie")))
    parity.compare_stats(sub, {k: gpu[k][ok] for k in ("conf", "entropy", "ent_norm", "gap", "argmax")})
    for b in range(len(cu) - 1):
        if b == bad_seq or res.flag_accept[b] or res.flag_lbs[b]:
            continue
        sl = slice(int(cu[b]), int(cu[b + 1]))
        for k in ("accepted", "tokens", "mask", "in_block"):
            assert np.array_equal(np.asarray(gpu[k][sl], np.int64),
                                  np.asarray(getattr(res, k)[sl], np.int64)), (k, b)
        assert np.array_equal(gpu["blk_meta"][b], res.blk_meta[b]), b
