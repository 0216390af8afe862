"""Dual-cache attention and the prefix-cache append on commit (Sec. 6.3) on
the GPU through the C ABI, against the oracle.

* Attention with a cached suffix range: tiny, LLaDA-8B and Dream-7B head
  shapes; empty, ragged and multi-tile suffixes, different per sequence.
* The append: after a step with kv_append = 1 the cache equals the oracle's
  kv_append of the pre-step cache with the step's final mask, bit for bit,
  on the device and the host-buffer entry points; the attention output of
  that step is the one without the append.
* The generation loop with a dual cache, step by step against the oracle's
  loop; and with a prefix cache that starts with the prompt only, so that
  the attention matches the oracle only if every committed row was
  appended."""
import dataclasses

import numpy as np
import pytest

import synth
from oracle import ebd_oracle as o
from tests import parity

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


def _with_suffix_cache(inp, extra, seed):
    """inp with a cache of prefix + extra positions; the positions after the
    prefix hold random K/V (those of the window's own positions are never
    read)."""
    sh = inp.shape
    rng = np.random.default_rng(seed)
    B, P = inp.k_cache.shape[0], inp.k_cache.shape[1]
    shape = (B, extra, sh.n_heads_kv, sh.head_dim)
    ke = synth.f32_to_bf16_bits(rng.standard_normal(shape).astype(np.float32))
    ve = synth.f32_to_bf16_bits(rng.standard_normal(shape).astype(np.float32))
    return dataclasses.replace(inp, k_cache=np.concatenate([inp.k_cache, ke], axis=1),
                               v_cache=np.concatenate([inp.v_cache, ve], axis=1))


def _attention(inp, suffix):
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    h = rt.Handle(rt.config_for(inp.shape, max_prefix=inp.k_cache.shape[1]))
    try:
        ds = rt.DeviceStep(inp, rt.DeviceWeights(w_lm=torch.zeros(8, dtype=torch.int16, device="cuda"),
                                                 w_emb=None, layout=0), outputs=False)
        a = ds.args()
        sfx = None
        if suffix is not None:
            sfx = torch.from_numpy(np.ascontiguousarray(suffix, np.int32)).cuda()
            a.suffix = sfx.data_ptr()
        E.check(E.ebd_attention(h.h, a, rt.stream_handle(None)), h.h)
        assert h.sync_status() == 0, E.ebd_last_error(h.h)
        return ds.fetch()["attn_out"]
    finally:
        h.close()


@pytest.mark.parametrize("S", [0, 1, 63, 64, 65, 200])
def test_suffix_tiny(S):
    sh = synth.tiny
    inp = _with_suffix_cache(synth.make_step_inputs(sh, weights=False), 32 + 200, seed=S)
    w = int(inp.cu_rows[1])
    suffix = np.array([[sh.prefix + w, S]], np.int32)
    got = _attention(inp, suffix)
    ref = o.window_attention(inp.q, inp.k_win, inp.v_win, inp.k_cache, inp.v_cache,
                             inp.cu_rows, inp.prefix_len, suffix)
    parity._close(f"attn S={S}", got, ref)


def test_suffix_llada_head_shape():
    """LLaDA-8B heads (32 x 128, MHA), prefix 512, window 32, suffix 480 (the
    rest of a 512-token response)."""
    sh = synth.llada
    inp = _with_suffix_cache(synth.make_step_inputs(sh, weights=False), 32 + 480, seed=11)
    suffix = np.array([[sh.prefix + 32, 480]], np.int32)
    got = _attention(inp, suffix)
    ref = o.window_attention(inp.q, inp.k_win, inp.v_win, inp.k_cache, inp.v_cache,
                             inp.cu_rows, inp.prefix_len, suffix)
    parity._close("attn llada dual", got, ref)


def test_suffix_dream_gqa_ragged():
    """Dream-7B heads (GQA 28 / 4), 8 sequences with windows of 16..64 rows,
    each with its own suffix length (0 for one of them)."""
    sh = synth.dream
    inp = _with_suffix_cache(synth.make_step_inputs(sh, weights=False), 64 + 300, seed=12)
    B = len(inp.cu_rows) - 1
    S = [0, 300, 17, 64, 129, 1, 250, 64][:B]
    suffix = np.array([[int(inp.prefix_len[b]) + int(inp.cu_rows[b + 1] - inp.cu_rows[b]), S[b]]
                       for b in range(B)], np.int32)
    got = _attention(inp, suffix)
    ref = o.window_attention(inp.q, inp.k_win, inp.v_win, inp.k_cache, inp.v_cache,
                             inp.cu_rows, inp.prefix_len, suffix)
    parity._close("attn dream dual", got, ref)


def _step_with_append(inp, host=False):
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    sh = inp.shape
    w = rt.upload_weights(inp)
    h = rt.Handle(rt.config_for(sh, max_prefix=inp.k_cache.shape[1]), w.w_emb)
    try:
        ds = rt.DeviceStep(inp, w)
        a = ds.args()
        a.kv_append = 1
        if not host:
            E.check(E.ebd_step(h.h, a, rt.stream_handle(None)), h.h)
            assert h.sync_status() == 0, E.ebd_last_error(h.h)
            out = ds.fetch()
        else:
            R, B = inp.rows, len(inp.cu_rows) - 1
            hb = dict(cu_rows=inp.cu_rows.astype(np.int32), prefix_len=inp.prefix_len.astype(np.int32),
                      row_pos=inp.row_pos.astype(np.int32), hidden=inp.hidden, q=inp.q,
                      k_win=inp.k_win, v_win=inp.v_win, tokens=inp.tokens.astype(np.int32),
                      mask=inp.mask.astype(np.uint8), in_block=inp.in_block.astype(np.uint8),
                      blk_meta=inp.blk_meta.astype(np.int32),
                      attn_out=np.zeros((R, sh.n_heads_q, sh.head_dim), np.float32),
                      accepted=np.zeros(R, np.uint8))
            hb = {k: np.ascontiguousarray(v) for k, v in hb.items()}
            if host == "pinned":  # mapped buffers: results stored by the kernels themselves
                pinned = {k: torch.from_numpy(v.view(np.int16) if v.dtype == np.uint16 else v).pin_memory()
                          for k, v in hb.items()}
                hb = {k: t.numpy().view(hb[k].dtype) for k, t in pinned.items()}
            for k, v in hb.items():
                setattr(a, k, v.ctypes.data)
            for k in ("conf", "entropy", "ent_norm", "gap", "argmax", "lbs_logit", "lps_prob"):
                setattr(a, k, None)
            E.check(E.ebd_step_host(h.h, a, rt.stream_handle(None)), h.h)
            torch.cuda.synchronize()
            assert h.sync_status() == 0, E.ebd_last_error(h.h)
            out = dict(mask=hb["mask"], attn_out=hb["attn_out"])
        out["k_cache"] = ds.k_cache.cpu().numpy().view(np.uint16)
        out["v_cache"] = ds.v_cache.cpu().numpy().view(np.uint16)
        return out
    finally:
        h.close()


@pytest.mark.parametrize("host", [False, True, "pinned"])
def test_append_tiny_matches_oracle(host):
    sh = synth.tiny
    inp = _with_suffix_cache(synth.make_step_inputs(sh), 64, seed=21)
    out = _step_with_append(inp, host=host)
    assert out["mask"].sum() < inp.mask.sum(), "the step committed nothing"
    kc, vc = o.kv_append(inp.k_cache, inp.v_cache, inp.k_win, inp.v_win, inp.cu_rows,
                         inp.row_pos, out["mask"])
    np.testing.assert_array_equal(out["k_cache"], kc)
    np.testing.assert_array_equal(out["v_cache"], vc)
    # the step's attention read the cache before the append
    ref = o.window_attention(inp.q, inp.k_win, inp.v_win, inp.k_cache, inp.v_cache,
                             inp.cu_rows, inp.prefix_len)
    parity._close("attn with append", out["attn_out"], ref)


def test_append_dream_batch():
    """8 sequences: every sequence's committed rows land in its own cache."""
    sh = synth.dream
    inp = synth.make_step_inputs(sh)
    inp = _with_suffix_cache(inp, 64, seed=22)
    out = _step_with_append(inp)
    kc, vc = o.kv_append(inp.k_cache, inp.v_cache, inp.k_win, inp.v_win, inp.cu_rows,
                         inp.row_pos, out["mask"])
    np.testing.assert_array_equal(out["k_cache"], kc)
    np.testing.assert_array_equal(out["v_cache"], vc)


def _prm(sh):
    return o.DecisionParams(tau=sh.tau, tau_psi=sh.tau_psi, l_min=sh.l_min, l_b=sh.l_b,
                            g_max=sh.g_max, eos_id=sh.eos_id, lps_enabled=bool(sh.lps_enabled))


def _loop_against_oracle(cache, append):
    from paper_2609_16450_gb300 import loop as lp
    from paper_2609_16450_gb300 import runtime as rt
    sh = synth.loop_tiny
    inp = synth.make_step_inputs(sh)
    w = rt.upload_weights(inp)
    h = rt.Handle(lp.config_for_loop(sh), w.w_emb)
    try:
        res = lp.run_loop(h, sh, w, lambda s, p: synth.loop_window_inputs(sh, s, p),
                          lambda p: synth.loop_kv(sh, p), attention=True, cache=cache,
                          append=append)
    finally:
        h.close()
    W = o.weights_f64(synth.router_weights(sh.seed, sh.d_base, sh.gen_len))
    toks, steps, commits, recs = o.generation_loop(
        sh, W, _prm(sh), lambda s, p: synth.loop_window_inputs(sh, s, p),
        lambda p: synth.loop_kv(sh, p), inp.w_lm, inp.w_emb, attention=True, cache=cache)
    compared = 0
    for g, r in zip(res.records, recs):
        assert g.window == r["window"], (g.step, g.window, r["window"])
        parity._close(f"attn step {g.step}", g.attn_out, r["attn"])
        if r["flag"] or r["flag_lbs"]:
            break  # a near-tie decision: the runs may part from here
        assert np.array_equal(g.accepted, r["accepted"]), g.step
        compared += 1
    assert compared >= 1
    return res


def test_loop_dual_cache_matches_oracle():
    _loop_against_oracle("dual", append=True)


def test_loop_prefix_cache_filled_by_appends():
    """The cache starts with the prompt only: every later prefix key the
    attention reads was written by an append, and after the loop (all rows
    committed) the cache holds every position's K/V."""
    sh = synth.loop_tiny
    res = _loop_against_oracle("prefix", append=True)
    if res.steps and not np.any(res.tokens < 0):
        kk, vv = synth.loop_kv(sh, np.arange(sh.prefix + sh.gen_len, dtype=np.int32))
        np.testing.assert_array_equal(res.k_cache.view(np.uint16), kk)
        np.testing.assert_array_equal(res.v_cache.view(np.uint16), vv)
