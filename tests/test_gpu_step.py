"""GPU parity of the whole decoding step against the CPU oracle, called
through the C ABI (ebd_step / ebd_step_host)."""
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


_cache = {}


def _setup(sh):
    from paper_2609_16450_gb300 import runtime as rt
    key = sh.name
    if key not in _cache:
        _cache.clear()
        inp = synth.make_step_inputs(sh)
        w = rt.upload_weights(inp)
        h = rt.Handle(rt.config_for(sh), w.w_emb)
        _cache[key] = (inp, w, h)
    return _cache[key]


def _run(sh, inp, w, h, attention=True):
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    ds = rt.DeviceStep(inp, w, attention=attention)
    E.check(E.ebd_step(h.h, ds.args(), rt.stream_handle(None)), h.h)
    assert h.sync_status() == 0
    return ds.fetch()


def _oracle(sh, inp, attention=True):
    W = o.weights_f64(synth.router_weights(sh.seed, sh.d_base, sh.gen_len))
    return o.step(inp, W, _prm(sh), attention=attention)


def _check(sh, inp, gpu, res, attention=True):
    rep = parity.compare_stats(res.stats, gpu)
    if attention:
        rep["attn"] = parity._close("attn_out", gpu["attn_out"], res.attn_out)
    rep.update(parity.compare_decision(res, gpu, inp, _prm(sh)))
    return rep


@pytest.mark.parametrize("state", ["select", "inblock"])
def test_tiny_step(state):
    sh = synth.tiny
    inp, w, h = _setup(sh)
    inp = synth.make_step_inputs(sh, weights=True)
    if state == "inblock":
        synth.preset_in_block(inp, 20)
    gpu = _run(sh, inp, w, h)
    res = _oracle(sh, inp)
    rep = _check(sh, inp, gpu, res)
    print(state, rep)
    assert gpu["accepted"].sum() >= 1


@pytest.mark.parametrize("layout", ["rowmajor", "packed"])
def test_llada_step(layout):
    from paper_2609_16450_gb300 import runtime as rt
    sh = synth.llada
    inp, w, h = _setup(sh)
    if layout == "packed":
        w = rt.pack_weights(h, rt.DeviceWeights(w_lm=w.w_lm, w_emb=w.w_emb))
    for state in ("select", "inblock"):
        inp2 = synth.make_step_inputs(sh)
        if state == "inblock":
            synth.preset_in_block(inp2, 20)
        gpu = _run(sh, inp2, w, h)
        res = _oracle(sh, inp2)
        print(state, _check(sh, inp2, gpu, res))


def test_host_step_matches_device_step():
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    sh = synth.tiny
    inp, w, h = _setup(sh)
    dev = _run(sh, inp, w, h)
    R, Hq, D = inp.rows, sh.n_heads_q, sh.head_dim
    host = {k: np.zeros(R, np.float32) for k in ("conf", "entropy", "ent_norm", "gap",
                                                  "lbs_logit", "lps_prob")}
    host["argmax"] = np.zeros(R, np.int32)
    host["accepted"] = np.zeros(R, np.uint8)
    host["attn_out"] = np.zeros((R, Hq, D), np.float32)
    st = {"tokens": inp.tokens.copy(), "mask": inp.mask.copy(), "in_block": inp.in_block.copy(),
          "blk_meta": inp.blk_meta.copy()}
    ins = {"cu_rows": inp.cu_rows.astype(np.int32), "prefix_len": inp.prefix_len.astype(np.int32),
           "row_pos": inp.row_pos.astype(np.int32), "hidden": inp.hidden, "q": inp.q,
           "k_win": inp.k_win, "v_win": inp.v_win}
    a = E.ebd_step_args()
    a.batch, a.rows = sh.batch, R
    for k, v in {**ins, **st, **host}.items():
        setattr(a, k, np.ascontiguousarray(v).ctypes.data)
    kc = torch.from_numpy(inp.k_cache.view(np.int16)).cuda()
    vc = torch.from_numpy(inp.v_cache.view(np.int16)).cuda()
    a.k_cache, a.v_cache, a.w_lm = kc.data_ptr(), vc.data_ptr(), w.w_lm.data_ptr()
    E.check(E.ebd_step_host(h.h, a, rt.stream_handle(None)), h.h)
    assert h.sync_status() == 0
    for k in ("conf", "entropy", "gap", "argmax", "accepted", "lbs_logit", "lps_prob"):
        np.testing.assert_array_equal(host[k], dev[k], err_msg=k)
    np.testing.assert_array_equal(host["attn_out"], dev["attn_out"])
    for k in ("tokens", "mask", "in_block", "blk_meta"):
        np.testing.assert_array_equal(st[k], dev[k], err_msg=k)


def test_host_step_pinned_matches_device_step():
    """The same with pinned (device-mapped) host buffers, which ebd_step_host
    moves with one kernel each way instead of copies."""
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    sh = synth.tiny
    inp, w, h = _setup(sh)
    dev = _run(sh, inp, w, h)
    R, Hq, D = inp.rows, sh.n_heads_q, sh.head_dim
    pin = lambda x: torch.from_numpy(np.ascontiguousarray(x)).pin_memory()  # noqa: E731
    host = {k: pin(np.zeros(R, np.float32)) for k in ("conf", "entropy", "ent_norm", "gap",
                                                       "lbs_logit", "lps_prob")}
    host["argmax"] = pin(np.zeros(R, np.int32))
    host["accepted"] = pin(np.zeros(R, np.uint8))
    host["attn_out"] = pin(np.zeros((R, Hq, D), np.float32))
    st = {"tokens": pin(inp.tokens), "mask": pin(inp.mask), "in_block": pin(inp.in_block),
          "blk_meta": pin(inp.blk_meta)}
    ins = {"cu_rows": pin(inp.cu_rows.astype(np.int32)), "prefix_len": pin(inp.prefix_len.astype(np.int32)),
           "row_pos": pin(inp.row_pos.astype(np.int32)), "hidden": pin(inp.hidden.view(np.int16)),
           "q": pin(inp.q.view(np.int16)), "k_win": pin(inp.k_win.view(np.int16)),
           "v_win": pin(inp.v_win.view(np.int16))}
    a = E.ebd_step_args()
    a.batch, a.rows = sh.batch, R
    for k, v in {**ins, **st, **host}.items():
        setattr(a, k, v.data_ptr())
    kc = torch.from_numpy(inp.k_cache.view(np.int16)).cuda()
    vc = torch.from_numpy(inp.v_cache.view(np.int16)).cuda()
    a.k_cache, a.v_cache, a.w_lm = kc.data_ptr(), vc.data_ptr(), w.w_lm.data_ptr()
    E.check(E.ebd_step_host(h.h, a, rt.stream_handle(None)), h.h)
    assert h.sync_status() == 0
    for k in ("conf", "entropy", "gap", "argmax", "accepted", "lbs_logit", "lps_prob"):
        np.testing.assert_array_equal(host[k].numpy(), dev[k], err_msg=k)
    np.testing.assert_array_equal(host["attn_out"].numpy(), dev["attn_out"])
    for k in ("tokens", "mask", "in_block", "blk_meta"):
        np.testing.assert_array_equal(st[k].numpy(), dev[k], err_msg=k)


def test_weights_init_and_roundtrip():
    from paper_2609_16450_gb300 import _ebd as E
    sh = synth.tiny
    inp, w, h = _setup(sh)
    s, blob = E.ebd_export_weights(h.h)
    assert s == 0
    ref = synth.pack_blob(synth.router_weights(sh.seed, sh.d_base, sh.gen_len), sh.d_base,
                          sh.gen_len)
    np.testing.assert_array_equal(blob, ref)
    assert E.ebd_import_weights(h.h, blob) == 0
    s, blob2 = E.ebd_export_weights(h.h)
    np.testing.assert_array_equal(blob2, blob)


def _modified_router(sh, lbs_head=None, lps_head=None):
    wts = synth.router_weights(sh.seed, sh.d_base, sh.gen_len)
    if lbs_head is not None:
        wts["lbs.head.b"] = synth.f32_to_bf16_bits(np.array([lbs_head], np.float32))
    if lps_head is not None:
        wts["lps.head.b"] = synth.f32_to_bf16_bits(np.array([lps_head], np.float32))
    return wts


@pytest.mark.parametrize("lbs_head,lps_head", [(4.0, 4.0), (-4.0, -4.0), (4.0, -4.0)])
def test_router_branches(lbs_head, lps_head):
    """Head biases of +-4 drive the LBS candidate set and the LPS accept rule
    through both outcomes; GPU and oracle use the same imported weights."""
    from paper_2609_16450_gb300 import _ebd as E
    sh = synth.tiny
    inp, w, h = _setup(sh)
    wts = _modified_router(sh, lbs_head, lps_head)
    assert E.ebd_import_weights(h.h, synth.pack_blob(wts, sh.d_base, sh.gen_len)) == 0
    try:
        inp2 = synth.make_step_inputs(sh)
        gpu = _run(sh, inp2, w, h)
        res = o.step(inp2, o.weights_f64(wts), _prm(sh))
        rep = _check(sh, inp2, gpu, res)
        print(lbs_head, lps_head, rep, gpu["accepted"].sum())
    finally:
        base = synth.pack_blob(synth.router_weights(sh.seed, sh.d_base, sh.gen_len), sh.d_base,
                               sh.gen_len)
        assert E.ebd_import_weights(h.h, base) == 0


def test_eos_removal():
    """Masked rows whose hidden state points at W_lm[eos] predict EOS and are
    removed from the LBS candidates."""
    sh = synth.tiny
    inp, w, h = _setup(sh)
    inp2 = synth.make_step_inputs(sh)
    eos_row = synth.bf16_to_f32(inp2.w_lm[sh.eos_id])
    masked = np.flatnonzero(inp2.mask)[:6]
    hid = synth.bf16_to_f32(inp2.hidden).reshape(inp2.rows, -1).copy()
    hid[masked] = eos_row / np.linalg.norm(eos_row) * 400.0
    inp2.hidden = synth.f32_to_bf16_bits(hid)
    wts = _modified_router(sh, lbs_head=4.0)
    from paper_2609_16450_gb300 import _ebd as E
    assert E.ebd_import_weights(h.h, synth.pack_blob(wts, sh.d_base, sh.gen_len)) == 0
    try:
        gpu = _run(sh, inp2, w, h)
        res = o.step(inp2, o.weights_f64(wts), _prm(sh))
        assert np.all(res.stats.argmax[masked] == sh.eos_id)
        _check(sh, inp2, gpu, res)
        assert np.all(gpu["argmax"][masked] == sh.eos_id)
    finally:
        base = synth.pack_blob(synth.router_weights(sh.seed, sh.d_base, sh.gen_len), sh.d_base,
                               sh.gen_len)
        assert E.ebd_import_weights(h.h, base) == 0


def test_timeout_is_reported_and_context_survives():
    """A bounded device-side wait that nothing completes gives EBD_ERR_TIMEOUT;
    the context stays usable afterwards."""
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    sh = synth.tiny
    inp, w, h = _setup(sh)
    hb = rt.Handle(rt.config_for(sh, debug_flags=E.EBD_DEBUG_FORCE_TIMEOUT), w.w_emb)
    ds = rt.DeviceStep(inp, w)
    E.check(E.ebd_step(hb.h, ds.args(), rt.stream_handle(None)), hb.h)
    assert hb.sync_status() == E.EBD_ERR_TIMEOUT
    hb.close()
    gpu = _run(sh, inp, w, h)
    res = _oracle(sh, inp)
    _check(sh, inp, gpu, res)


def test_copy_stream_timeout_is_reported_and_context_survives():
    """ebd_step_host from pinned buffers: q and the window K/V come in on the
    copy stream and the attention waits, time-limited, for its ticket.  A
    ticket that never comes gives EBD_ERR_TIMEOUT; the context stays usable."""
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    sh = synth.tiny
    inp, w, h = _setup(sh)
    hb = rt.Handle(rt.config_for(sh, debug_flags=E.EBD_DEBUG_FORCE_COPY_TIMEOUT), w.w_emb)
    ds = rt.DeviceStep(inp, w)
    host, a = _pinned_host_args(sh, inp, ds, w)
    E.check(E.ebd_step_host(hb.h, a, rt.stream_handle(None)), hb.h)
    assert hb.sync_status() == E.EBD_ERR_TIMEOUT
    hb.close()
    gpu = _run(sh, inp, w, h)
    res = _oracle(sh, inp)
    _check(sh, inp, gpu, res)


def _pinned_host_args(sh, inp, ds, w):
    R = inp.rows
    pin = lambda a: torch.from_numpy(np.ascontiguousarray(a)).pin_memory()  # noqa: E731
    host = dict(cu_rows=pin(inp.cu_rows.astype(np.int32)), prefix_len=pin(inp.prefix_len.astype(np.int32)),
                row_pos=pin(inp.row_pos.astype(np.int32)), hidden=pin(inp.hidden.view(np.int16)),
                q=pin(inp.q.view(np.int16)), k_win=pin(inp.k_win.view(np.int16)),
                v_win=pin(inp.v_win.view(np.int16)), tokens=pin(inp.tokens.astype(np.int32)),
                mask=pin(inp.mask.astype(np.uint8)), in_block=pin(inp.in_block.astype(np.uint8)),
                blk_meta=pin(inp.blk_meta.astype(np.int32)),
                attn_out=torch.empty((R, sh.n_heads_q, sh.head_dim), dtype=torch.float32).pin_memory(),
                conf=torch.empty(R, dtype=torch.float32).pin_memory(),
                argmax=torch.empty(R, dtype=torch.int32).pin_memory(),
                accepted=torch.empty(R, dtype=torch.uint8).pin_memory())
    from paper_2609_16450_gb300 import _ebd as E
    a = E.ebd_step_args()
    a.batch, a.rows = sh.batch, R
    for k, t in host.items():
        setattr(a, k, t.data_ptr())
    a.k_cache, a.v_cache, a.w_lm = ds.k_cache.data_ptr(), ds.v_cache.data_ptr(), w.w_lm.data_ptr()
    a.w_lm_layout = w.layout
    return host, a


def test_host_step_captured_in_a_graph():
    """ebd_step_host captured into a CUDA graph (the capture takes the
    single-gather route) and replayed gives the uncaptured call's results."""
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    sh = synth.tiny
    inp, w, h = _setup(sh)
    ds = rt.DeviceStep(inp, w)
    host, a = _pinned_host_args(sh, inp, ds, w)
    st0 = {k: host[k].clone() for k in ("tokens", "mask", "in_block", "blk_meta")}
    stream = torch.cuda.Stream()
    E.check(E.ebd_step_host(h.h, a, stream.cuda_stream), h.h)
    stream.synchronize()
    assert h.sync_status() == 0
    ref = {k: t.clone() for k, t in host.items()}
    for k, v in st0.items():
        host[k].copy_(v)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        E.check(E.ebd_step_host(h.h, a, stream.cuda_stream), h.h)
    torch.cuda.synchronize()
    for k, v in st0.items():  # the capture ran nothing
        host[k].copy_(v)
    g.replay()
    torch.cuda.synchronize()
    assert h.sync_status() == 0
    for k in ("tokens", "mask", "in_block", "blk_meta", "argmax", "accepted"):
        assert torch.equal(host[k], ref[k]), k
    for k in ("conf", "attn_out"):
        assert torch.equal(host[k], ref[k]), k


def test_overlapped_and_serial_and_graph_steps_agree():
    """The production order (attention as a programmatic dependent of the
    decision), the fully serial order and a CUDA-graph replay give identical
    bits."""
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    sh = synth.tiny
    inp, w, h = _setup(sh)
    outs = []
    for mode in (0, 1, 2):
        E.check(E.ebd_profile_enable(h.h, mode), h.h)
        outs.append(_run(sh, inp, w, h))
    E.check(E.ebd_profile_enable(h.h, 0), h.h)
    ds = rt.DeviceStep(inp, w)
    args = ds.args()
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        E.check(E.ebd_step(h.h, args, stream.cuda_stream), h.h)
    torch.cuda.synchronize()
    ds.restore_state()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        E.check(E.ebd_step(h.h, args, stream.cuda_stream), h.h)
    torch.cuda.synchronize()
    ds.restore_state()
    for k in ("attn_out", "conf", "argmax"):
        ds_val = getattr(ds, k)
        ds_val.zero_()
    torch.cuda.synchronize()
    g.replay()
    torch.cuda.synchronize()
    assert h.sync_status() == 0
    outs.append(ds.fetch())
    for o2 in outs[1:]:
        for k in outs[0]:
            np.testing.assert_array_equal(outs[0][k], o2[k], err_msg=k)
