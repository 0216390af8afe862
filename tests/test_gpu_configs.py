"""GPU parity on the Dream-7B shaped step and on points of the throughput
sweep, through the C ABI.  At these sizes the oracle's full logits rows take
minutes, so:
  * the window attention is compared in full (Dream) or on sampled sequences;
  * the statistics are compared on sampled rows (first, middle and last row
    of every sequence, at most 48 rows) and, for Dream, on every masked row
    of its shortest and its longest sequence;
  * the decision is compared with the GPU's statistics fed to the oracle's
    decision (bit-exact apart from sequences flagged for a near-tie), which
    checks the routers, the filters and the commit at full size."""
import numpy as np
import pytest

import synth
from oracle import ebd_oracle as o
from tests import parity

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


def _prm(sh):
    return o.DecisionParams(tau=sh.tau, tau_psi=sh.tau_psi, l_min=sh.l_min, l_b=sh.l_b,
                            g_max=sh.g_max, eos_id=sh.eos_id, lps_enabled=bool(sh.lps_enabled))


def _gpu_step(sh, inp, h, w):
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    ds = rt.DeviceStep(inp, w)
    E.check(E.ebd_step(h.h, ds.args(), rt.stream_handle(None)), h.h)
    assert h.sync_status() == 0, E.ebd_last_error(h.h)
    return ds.fetch()


def _sample_rows(cu_rows, cap=48):
    rows = []
    for b in range(len(cu_rows) - 1):
        r0, r1 = int(cu_rows[b]), int(cu_rows[b + 1])
        rows += sorted({r0, (r0 + r1) // 2, r1 - 1})
    rows = np.array(sorted(set(rows)), dtype=np.int64)
    if rows.size > cap:
        rows = rows[np.linspace(0, rows.size - 1, cap).astype(np.int64)]
    return rows


def _whole_sequences(inp, seqs):
    """Every masked row of the given sequences."""
    rows = []
    for b in seqs:
        r0, r1 = int(inp.cu_rows[b]), int(inp.cu_rows[b + 1])
        rows += [r for r in range(r0, r1) if inp.mask[r]]
    return rows


def _check_stats_sampled(inp, gpu, whole=()):
    rows = np.array(sorted(set(_sample_rows(inp.cu_rows).tolist()) |
                           set(_whole_sequences(inp, whole))), dtype=np.int64)
    st = o.softmax_stats(o.lm_logits(inp.hidden.reshape(inp.rows, -1)[rows],
                                     inp.w_lm.reshape(inp.shape.vocab, -1)))
    return parity.compare_stats(st, {k: gpu[k][rows] for k in
                                     ("conf", "entropy", "ent_norm", "gap", "argmax")})


def _check_attention(inp, gpu, seqs):
    sh = inp.shape
    for b in seqs:
        r0, r1 = int(inp.cu_rows[b]), int(inp.cu_rows[b + 1])
        ref = o.window_attention(inp.q[r0:r1], inp.k_win[r0:r1], inp.v_win[r0:r1],
                                 inp.k_cache[b:b + 1], inp.v_cache[b:b + 1],
                                 np.array([0, r1 - r0]), inp.prefix_len[b:b + 1])
        parity._close(f"attn_out[{b}]", gpu["attn_out"][r0:r1], ref)


def _check_decision_injected(inp, gpu, sh):
    """The oracle's decision on the GPU's statistics."""
    R = inp.rows
    st = o.RowStats(conf=gpu["conf"].astype(np.float64), entropy=gpu["entropy"].astype(np.float64),
                    ent_norm=gpu["ent_norm"].astype(np.float64),
                    gap=gpu["gap"].astype(np.float64), argmax=gpu["argmax"].astype(np.int64),
                    logit_gap=np.full(R, np.inf), near_tie=np.zeros(R, bool))
    W = o.weights_f64(synth.router_weights(sh.seed, sh.d_base, sh.gen_len))
    res = o.decide(inp.cu_rows, inp.row_pos, inp.tokens, inp.mask, inp.in_block, inp.blk_meta,
                   st, inp.w_emb, W, _prm(sh))
    return parity.compare_decision(res, gpu, inp, _prm(sh))


_cache = {}


def _setup(sh, packed=True):
    from paper_2609_16450_gb300 import runtime as rt
    if sh.name not in _cache:
        _cache.clear()
        inp = synth.make_step_inputs(sh)
        w = rt.upload_weights(inp)
        h = rt.Handle(rt.config_for(sh), w.w_emb)
        if packed:
            w = rt.pack_weights(h, w)
        _cache[sh.name] = (inp, w, h)
    return _cache[sh.name]


@pytest.mark.parametrize("state", ["select", "inblock"])
def test_dream_step(state):
    sh = synth.dream
    inp0, w, h = _setup(sh)
    inp = synth.make_step_inputs(sh, weights=False)
    inp.w_lm, inp.w_emb = inp0.w_lm, inp0.w_emb
    if state == "inblock":
        synth.preset_in_block(inp, 20)
    gpu = _gpu_step(sh, inp, h, w)
    # every masked row of the shortest and the longest sequence, and the
    # first, middle and last row of every other
    lens = np.diff(inp.cu_rows)
    rep = {"stats": _check_stats_sampled(inp, gpu, whole=(int(np.argmin(lens)), int(np.argmax(lens))))}
    _check_attention(inp, gpu, range(sh.batch))
    rep["decision"] = _check_decision_injected(inp, gpu, sh)
    print(state, rep)
    # every sequence with masked rows commits at least one of them
    for b in range(sh.batch):
        r0, r1 = int(inp.cu_rows[b]), int(inp.cu_rows[b + 1])
        if inp.mask[r0:r1].any():
            assert gpu["accepted"][r0:r1].sum() >= 1


@pytest.mark.parametrize("point", [(4, 1024, 32), (16, 256, 64), (1, 4096, 8), (64, 1024, 64), (64, 4096, 64)])
def test_sweep_point(point):
    sh = synth.sweep_point(*point)
    inp, w, h = _setup(sh)
    gpu = _gpu_step(sh, inp, h, w)
    rep = {"stats": _check_stats_sampled(inp, gpu)}
    _check_attention(inp, gpu, sorted({0, sh.batch - 1}))
    rep["decision"] = _check_decision_injected(inp, gpu, sh)
    print(point, rep)
