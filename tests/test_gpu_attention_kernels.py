"""Both window-attention kernels -- tcgen05 (128-row query tiles, S and O in
TMEM) and mma.sync (64-row tiles) -- against the oracle's
softmax(Q K^T / sqrt(D)) V through ebd_attention, each forced in turn with
EBD_ATTN_KERNEL (Sec. 3: bidirectional attention over the cached prefix and
the window; Sec. 6.3: prefix and dual cache).

* tiny heads (4 x 64) with and without a cached suffix;
* LLaDA-8B heads (32 x 128, MHA) at prefix 512, window 32 (key splits and
  their merge), with and without a 480-key suffix;
* Dream-7B heads (GQA 28 / 4, up to 448 query rows per kv head: several
  query tiles), ragged windows, a suffix per sequence;
* degenerate windows: no prefix, one row, splits that get no key chunk;
* 64-dim heads with GQA 8 / 2 at the query-tile boundaries (64, 65, 128 and 4
  query rows per kv head) and ragged;
* sixteen sequences (one split per tile) and a long prefix (4096);
* the key range forced into 3 and 8 splits per query tile;
* scores that grow from chunk to chunk by far more than the tcgen05 kernel's
  rescale threshold (the running maximum moves, O is rescaled in TMEM), that
  shrink (it never moves), and a dominant key per row (probabilities near 1,
  where the high/low split of P matters)."""
import dataclasses

import numpy as np
import pytest

import synth
from oracle import ebd_oracle as o
from tests import parity
from tests.test_gpu_dual_cache import _attention, _with_suffix_cache

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(params=["tc", "mma"])
def kernel(request, monkeypatch):
    monkeypatch.setenv("EBD_ATTN_KERNEL", request.param)
    return request.param


def _ref(inp, suffix=None):
    return o.window_attention(inp.q, inp.k_win, inp.v_win, inp.k_cache, inp.v_cache,
                              inp.cu_rows, inp.prefix_len, suffix)


def _check(name, inp, suffix=None):
    got = _attention(inp, suffix)
    parity._close(name, got, _ref(inp, suffix))
    return got


@pytest.mark.parametrize("S", [0, 65])
def test_tiny(kernel, S):
    sh = synth.tiny
    inp = _with_suffix_cache(synth.make_step_inputs(sh, weights=False), 32 + 100, seed=3 + S)
    w = int(inp.cu_rows[1])
    suffix = np.array([[sh.prefix + w, S]], np.int32) if S else None
    _check(f"tiny S={S}", inp, suffix)


@pytest.mark.parametrize("dual", [False, True])
def test_llada_heads(kernel, dual):
    sh = synth.llada
    inp = synth.make_step_inputs(sh, weights=False)
    suffix = None
    if dual:
        inp = _with_suffix_cache(inp, 32 + 480, seed=21)
        suffix = np.array([[sh.prefix + 32, 480]], np.int32)
    _check(f"llada dual={dual}", inp, suffix)


def test_dream_gqa_ragged(kernel):
    sh = synth.dream
    inp = _with_suffix_cache(synth.make_step_inputs(sh, weights=False), 64 + 200, seed=22)
    B = len(inp.cu_rows) - 1
    S = [0, 200, 17, 64, 129, 1, 150, 64][:B]
    suffix = np.array([[int(inp.prefix_len[b]) + int(inp.cu_rows[b + 1] - inp.cu_rows[b]), S[b]]
                       for b in range(B)], np.int32)
    _check("dream", inp, suffix)


def test_degenerate_windows(kernel):
    """Windows of 0, 1, 64, 7, 20 and 33 rows; prefixes of 128, 0, 128, 5,
    64 and 1 keys (with a cache of 128 positions the key range splits into
    up to 3 parts, so short sequences leave splits without a chunk)."""
    sh = synth.tiny.with_(name="attn_edge", batch=6, windows=(0, 1, 64, 7, 20, 33), seed=23)
    inp = synth.make_step_inputs(sh, weights=False,
                                 prefix_lens=np.array([128, 0, 128, 5, 64, 1]))
    got = _check("degenerate", inp)
    assert got.shape[0] == int(inp.cu_rows[-1])


def test_sixteen_sequences(kernel):
    sh = synth.sweep_point(16, 256, 8)
    _check("16 x 256 x 8", synth.make_step_inputs(sh, weights=False))


def test_long_prefix(kernel):
    sh = synth.sweep_point(4, 4096, 32).with_(name="attn_long", batch=2, windows=(32, 32))
    _check("2 x 4096 x 32", synth.make_step_inputs(sh, weights=False))


def _scaled_cache(inp, f):
    """K cache rows at position t multiplied by f(t) (bf16 bits again)."""
    k = synth.bf16_to_f32(inp.k_cache)
    t = np.arange(k.shape[1], dtype=np.float32)
    k = k * f(t)[None, :, None, None].astype(np.float32)
    return dataclasses.replace(inp, k_cache=synth.f32_to_bf16_bits(k))


@pytest.mark.parametrize("trend", ["growing", "shrinking"])
def test_running_maximum(kernel, trend):
    """Prefix 512 at LLaDA-8B heads with the key norms ramped over the
    prefix: growing, each 64-key chunk's maximum score exceeds the last by
    several units (in log2), so the running maximum moves at every chunk;
    shrinking, the first chunk holds it."""
    sh = synth.llada
    inp = synth.make_step_inputs(sh, weights=False)
    ramp = (lambda t: 0.25 + t / 64.0) if trend == "growing" else (lambda t: 8.25 - t / 64.0)
    _check(trend, _scaled_cache(inp, ramp))


def test_dominant_key(kernel):
    """One cached key per query row equal to 12 / sqrt(D) x its query: that
    key takes almost all of the probability (p close to 1), so P V is exact
    only with the probabilities' low part."""
    sh = synth.tiny
    inp = synth.make_step_inputs(sh, weights=False)
    q = synth.bf16_to_f32(inp.q)          # [R][Hq][D]
    k = synth.bf16_to_f32(inp.k_cache)    # [B][P][Hkv][D]
    R = q.shape[0]
    for r in range(R):
        k[0, (7 * r) % k.shape[1], :, :] = 12.0 * q[r, :, :] / np.sqrt(sh.head_dim)
    inp = dataclasses.replace(inp, k_cache=synth.f32_to_bf16_bits(k))
    got = _check("dominant", inp)
    assert np.all(np.isfinite(got))


@pytest.mark.parametrize("splits", [3, 8])
def test_key_splits(kernel, monkeypatch, splits):
    """The key range split over several CTAs per query tile (the last CTA of a
    tile combines their partial maxima, sums and outputs): LLaDA-8B heads at
    prefix 512, and the degenerate windows, where short sequences leave some
    splits without a key chunk."""
    monkeypatch.setenv("EBD_ATTN_SPLITS", str(splits))
    _check(f"llada splits={splits}", synth.make_step_inputs(synth.llada, weights=False))
    sh = synth.tiny.with_(name="attn_edge", batch=6, windows=(0, 1, 64, 7, 20, 33), seed=23)
    inp = synth.make_step_inputs(sh, weights=False, prefix_lens=np.array([128, 0, 128, 5, 64, 1]))
    _check(f"degenerate splits={splits}", inp)


@pytest.mark.parametrize("windows", [(32, 33, 64, 1), (31, 17, 48, 40)])
def test_gqa_tile_boundaries(kernel, windows):
    """64-dim heads with GQA 8 / 2 (4 query heads per kv head): windows of
    32, 33, 64 and 1 rows give 128, 132, 256 and 4 query rows per kv head,
    i.e. tiles of exactly 64 rows, a tile of 4 after two full ones, and a
    lone short tile (the tcgen05 kernel repeats 32- and 64-row tiles over
    its lane quadrants differently); the second set is ragged throughout."""
    sh = synth.tiny.with_(name="attn_gqa", batch=len(windows), windows=windows,
                          n_heads_q=8, n_heads_kv=2, seed=31)
    inp = synth.make_step_inputs(sh, weights=False,
                                 prefix_lens=np.array([128, 77, 0, 128][:len(windows)]))
    _check(f"gqa {windows}", inp)
