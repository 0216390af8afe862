"""Pins of the oracle's window attention (no GPU): a library routine
(torch's scaled_dot_product_attention in float64), and closed forms (one key
gives its value, identical keys give the mean value, zero queries give the
mean), plus the masking structure (ragged prefixes, batch separation, GQA
head mapping)."""
import numpy as np
import pytest
import torch

import synth
from oracle import ebd_oracle as o


def _bits(x):
    return synth.f32_to_bf16_bits(np.asarray(x, np.float32))


def _case(B=2, w=(3, 5), P=7, Hq=4, Hkv=2, D=8, seed=0):
    rng = np.random.default_rng(seed)
    R = sum(w)
    cu = np.concatenate([[0], np.cumsum(w)]).astype(np.int32)
    q = _bits(rng.standard_normal((R, Hq, D)))
    kw = _bits(rng.standard_normal((R, Hkv, D)))
    vw = _bits(rng.standard_normal((R, Hkv, D)))
    kc = _bits(rng.standard_normal((B, P, Hkv, D)))
    vc = _bits(rng.standard_normal((B, P, Hkv, D)))
    return q, kw, vw, kc, vc, cu


def test_matches_torch_sdpa():
    q, kw, vw, kc, vc, cu = _case()
    pl = np.array([7, 4], np.int32)
    out = o.window_attention(q, kw, vw, kc, vc, cu, pl)
    Hq, Hkv = q.shape[1], kw.shape[1]
    for b in range(2):
        r0, r1 = cu[b], cu[b + 1]
        for h in range(Hq):
            g = h // (Hq // Hkv)
            K = np.concatenate([o.bf16(kc[b, :pl[b], g]), o.bf16(kw[r0:r1, g])])
            V = np.concatenate([o.bf16(vc[b, :pl[b], g]), o.bf16(vw[r0:r1, g])])
            Q = o.bf16(q[r0:r1, h])
            ref = torch.nn.functional.scaled_dot_product_attention(
                torch.from_numpy(Q)[None], torch.from_numpy(K)[None],
                torch.from_numpy(V)[None])[0].numpy()
            np.testing.assert_allclose(out[r0:r1, h], ref, rtol=1e-12, atol=1e-12)


def test_single_key_returns_value():
    q, kw, vw, kc, vc, cu = _case(B=1, w=(1,), P=3, Hq=2, Hkv=2)
    out = o.window_attention(q, kw, vw, kc, vc, cu, np.array([0], np.int32))
    np.testing.assert_array_equal(out[0], o.bf16(vw[0]))


def test_identical_keys_give_mean_value_and_zero_query_too():
    q, kw, vw, kc, vc, cu = _case(B=1, w=(4,), P=6, Hq=2, Hkv=1)
    kc[:] = kc[0, 0]
    kw[:] = kc[0, 0]
    out = o.window_attention(q, kw, vw, kc, vc, cu, np.array([6], np.int32))
    allv = np.concatenate([o.bf16(vc[0, :, 0]), o.bf16(vw[:, 0])])
    np.testing.assert_allclose(out[:, 0], np.broadcast_to(allv.mean(0), out[:, 0].shape), atol=1e-12)
    q2, kw2, vw2, kc2, vc2, cu2 = _case(B=1, w=(4,), P=6, Hq=2, Hkv=1, seed=3)
    q2[:] = 0
    out2 = o.window_attention(q2, kw2, vw2, kc2, vc2, cu2, np.array([6], np.int32))
    allv2 = np.concatenate([o.bf16(vc2[0, :, 0]), o.bf16(vw2[:, 0])])
    np.testing.assert_allclose(out2[:, 1], np.broadcast_to(allv2.mean(0), out2[:, 1].shape), atol=1e-12)


def test_ragged_prefix_and_batch_separation():
    """A huge-score key beyond prefix_len, or in the other sequence's window,
    must not be attended to."""
    D = 8
    q, kw, vw, kc, vc, cu = _case(B=2, w=(2, 2), P=5, Hq=1, Hkv=1, D=D)
    q[:] = _bits(np.ones((4, 1, D)))
    kc[0, 4] = _bits(np.full((1, D), 30.0))       # beyond prefix_len[0] = 4
    vc[0, 4] = _bits(np.full((1, D), 512.0))
    kw[2:] = _bits(np.full((2, 1, D), 30.0))       # sequence 1's window keys
    vw[2:] = _bits(np.full((2, 1, D), -512.0))
    out = o.window_attention(q, kw, vw, kc, vc, cu, np.array([4, 5], np.int32))
    assert np.all(np.abs(out[:2]) < 10)            # sequence 0 ignores both
    np.testing.assert_allclose(out[2:], -512.0, atol=1e-6)  # sequence 1 sees its own


def test_gqa_head_mapping():
    D = 4
    q, kw, vw, kc, vc, cu = _case(B=1, w=(1,), P=0, Hq=4, Hkv=2, D=D)
    vw[0, 0] = _bits(np.full(D, 1.0))
    vw[0, 1] = _bits(np.full(D, 2.0))
    out = o.window_attention(q, kw, vw, kc[:, :0], vc[:, :0], cu, np.array([0], np.int32))
    assert out[0, :, 0].tolist() == [1.0, 1.0, 2.0, 2.0]


# ---------------------------------------------------------------- dual cache
def test_suffix_matches_torch_sdpa():
    """Suffix keys (dual cache) against the library routine on the keys
    prefix ++ window ++ cache[s0:s0+S]."""
    q, kw, vw, kc, vc, cu = _case(B=2, w=(3, 5), P=12)
    pl = np.array([4, 2], np.int32)
    sfx = np.array([[7, 5], [9, 3]], np.int32)
    out = o.window_attention(q, kw, vw, kc, vc, cu, pl, sfx)
    Hq, Hkv = q.shape[1], kw.shape[1]
    for b in range(2):
        r0, r1 = cu[b], cu[b + 1]
        s0, S = sfx[b]
        for h in range(Hq):
            g = h // (Hq // Hkv)
            K = np.concatenate([o.bf16(kc[b, :pl[b], g]), o.bf16(kw[r0:r1, g]), o.bf16(kc[b, s0:s0 + S, g])])
            V = np.concatenate([o.bf16(vc[b, :pl[b], g]), o.bf16(vw[r0:r1, g]), o.bf16(vc[b, s0:s0 + S, g])])
            ref = torch.nn.functional.scaled_dot_product_attention(
                torch.from_numpy(o.bf16(q[r0:r1, h]))[None], torch.from_numpy(K)[None],
                torch.from_numpy(V)[None])[0].numpy()
            np.testing.assert_allclose(out[r0:r1, h], ref, rtol=1e-12, atol=1e-12)


def test_empty_suffix_is_the_prefix_cache():
    q, kw, vw, kc, vc, cu = _case(B=2, w=(3, 5), P=9)
    pl = np.array([6, 3], np.int32)
    a = o.window_attention(q, kw, vw, kc, vc, cu, pl)
    b = o.window_attention(q, kw, vw, kc, vc, cu, pl, np.array([[7, 0], [4, 0]], np.int32))
    np.testing.assert_array_equal(a, b)


def test_suffix_keys_count_once_in_any_order():
    """Softmax attention does not depend on the order of the keys: moving the
    suffix range to the end of the prefix (and growing prefix_len) must give
    the same output.  A wrong offset, a lost or doubled segment, or keys and
    values taken from different positions break it."""
    q, kw, vw, kc, vc, cu = _case(B=2, w=(4, 2), P=16, seed=5)
    pl = np.array([5, 3], np.int32)
    sfx = np.array([[9, 6], [11, 4]], np.int32)
    out = o.window_attention(q, kw, vw, kc, vc, cu, pl, sfx)
    kc2, vc2 = kc.copy(), vc.copy()
    pl2 = pl.copy()
    for b in range(2):
        s0, S = sfx[b]
        kc2[b, pl[b]:pl[b] + S] = kc[b, s0:s0 + S]
        vc2[b, pl[b]:pl[b] + S] = vc[b, s0:s0 + S]
        pl2[b] = pl[b] + S
    ref = o.window_attention(q, kw, vw, kc2, vc2, cu, pl2)
    np.testing.assert_allclose(out, ref, rtol=1e-12, atol=1e-12)


def test_kv_append_writes_committed_rows_only():
    """Committed rows (mask 0) land at their positions bit for bit; masked
    rows, other positions, other sequences and out-of-range positions are
    untouched; appending twice is appending once."""
    q, kw, vw, kc, vc, cu = _case(B=2, w=(3, 4), P=10, seed=7)
    row_pos = np.array([2, 3, 4, 5, 6, 7, 12], np.int32)   # the last one is outside the cache
    mask = np.array([0, 1, 0, 0, 0, 1, 0], np.uint8)
    kc2, vc2 = o.kv_append(kc, vc, kw, vw, cu, row_pos, mask)
    touched = {(0, 2): 0, (0, 4): 2, (1, 5): 3, (1, 6): 4}
    for b in range(2):
        for pos in range(10):
            if (b, pos) in touched:
                r = touched[(b, pos)]
                np.testing.assert_array_equal(kc2[b, pos], kw[r])
                np.testing.assert_array_equal(vc2[b, pos], vw[r])
            else:
                np.testing.assert_array_equal(kc2[b, pos], kc[b, pos])
                np.testing.assert_array_equal(vc2[b, pos], vc[b, pos])
    kc3, vc3 = o.kv_append(kc2, vc2, kw, vw, cu, row_pos, mask)
    np.testing.assert_array_equal(kc3, kc2)
    np.testing.assert_array_equal(vc3, vc2)
