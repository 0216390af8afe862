"""Seeded synthetic tensors for one decoding step.

Random numbers come from NumPy's Philox bit generator (Salmon et al., SC'11),
keyed by (seed, tensor id, chunk); chunks have a fixed size, so a tensor's
values do not depend on how many threads draw them.  Everything is rounded to
bf16 here, once, and both consumers read the same bytes.

Value recipe (stand-ins for the paper's LLaDA-8B / Dream-7B decoding runs):
  hidden[r]   = N(0,1) * s_r,  s_r = exp(U[ln lo, ln hi])  (mixed entropy)
  W_lm        ~ N(0, w_lm_std^2)
  W_e         ~ N(0, w_emb_std^2)            (frozen token embedding)
  q, K, V     ~ N(0, 1)
  mask        round(mask_frac * w_b) rows of each window, seeded permutation
  tokens      unmasked rows U[0, V); masked rows hold MASK_TOKEN
"""
from __future__ import annotations

import dataclasses
import math
import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass
from functools import lru_cache
from typing import Optional

import numpy as np

from .configs import Shape

MASK_TOKEN = -1
_CHUNK = 1 << 22

# tensor ids of the step inputs
T_WLM, T_WEMB, T_HID, T_HSCALE, T_Q, T_KWIN, T_VWIN, T_KC, T_VC = range(1, 10)
T_PERM, T_TOK, T_WIN, T_LOOPHID, T_LOOPQ, T_LOOPKV = range(10, 16)
T_KSUF, T_VSUF = range(16, 18)


def _gen(seed: int, tid: int, chunk: int) -> np.random.Generator:
    key = np.array([seed & 0xFFFFFFFFFFFFFFFF,
                    ((tid & 0xFFFFFFFF) << 32) | (chunk & 0xFFFFFFFF)],
                   dtype=np.uint64)
    return np.random.Generator(np.random.Philox(key=key))


def _threads() -> int:
    return max(1, min(32, os.cpu_count() or 1))


def normal_f32(seed: int, tid: int, n: int, std: float = 1.0) -> np.ndarray:
    """n standard normals (float32), scaled by std in float32."""
    out = np.empty(n, dtype=np.float32)
    nch = (n + _CHUNK - 1) // _CHUNK

    def fill(c):
        lo, hi = c * _CHUNK, min(n, (c + 1) * _CHUNK)
        _gen(seed, tid, c).standard_normal(out=out[lo:hi], dtype=np.float32)
        if std != 1.0:
            out[lo:hi] *= np.float32(std)

    if nch <= 1:
        for c in range(nch):
            fill(c)
    else:
        with ThreadPoolExecutor(_threads()) as ex:
            list(ex.map(fill, range(nch)))
    return out


def uniform01(seed: int, tid: int, n: int) -> np.ndarray:
    """n uniforms in [0, 1) (float64, 53-bit)."""
    return _gen(seed, tid, 0).random(n)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bf16 (round to nearest even); returns uint16 bits."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty(x.shape, dtype=np.uint16)
    flat_in = x.reshape(-1).view(np.uint32)
    flat_out = out.reshape(-1)
    n = flat_in.size

    def conv(c):
        lo, hi = c * _CHUNK, min(n, (c + 1) * _CHUNK)
        u = flat_in[lo:hi].astype(np.uint64)
        u = u + np.uint64(0x7FFF) + ((u >> np.uint64(16)) & np.uint64(1))
        flat_out[lo:hi] = (u >> np.uint64(16)).astype(np.uint16)

    nch = (n + _CHUNK - 1) // _CHUNK
    if nch <= 1:
        for c in range(nch):
            conv(c)
    else:
        with ThreadPoolExecutor(_threads()) as ex:
            list(ex.map(conv, range(nch)))
    return out


def bf16_to_f32(b: np.ndarray) -> np.ndarray:
    b = np.ascontiguousarray(b, dtype=np.uint16)
    return (b.astype(np.uint32) << np.uint32(16)).view(np.float32)


def bf16_round(x: np.ndarray) -> np.ndarray:
    return bf16_to_f32(f32_to_bf16_bits(x))


def normal_bf16(seed: int, tid: int, shape, std: float = 1.0) -> np.ndarray:
    n = int(np.prod(shape))
    return f32_to_bf16_bits(normal_f32(seed, tid, n, std)).reshape(shape)


@lru_cache(maxsize=4)
def _big_weight(seed: int, tid: int, rows: int, cols: int, std: float):
    w = normal_bf16(seed, tid, (rows, cols), std)
    w.setflags(write=False)
    return w


@dataclass
class StepInputs:
    """Host tensors of one decoding step (bf16 tensors as uint16 bits)."""
    shape: Shape
    cu_rows: np.ndarray      # int32[B+1]
    prefix_len: np.ndarray   # int32[B]
    row_pos: np.ndarray      # int32[R], absolute position of each window row
    hidden: np.ndarray       # u16[R][d]
    q: np.ndarray            # u16[R][Hq][D]
    k_win: np.ndarray        # u16[R][Hkv][D]
    v_win: np.ndarray        # u16[R][Hkv][D]
    k_cache: np.ndarray      # u16[B][P][Hkv][D]
    v_cache: np.ndarray      # u16[B][P][Hkv][D]
    w_lm: np.ndarray         # u16[V][d]
    w_emb: np.ndarray        # u16[V][d_base]
    tokens: np.ndarray       # int32[R]
    mask: np.ndarray         # u8[R]
    in_block: np.ndarray     # u8[R]
    blk_meta: np.ndarray     # int32[B][2] = {b, |B|}

    @property
    def rows(self) -> int:
        return int(self.cu_rows[-1])

    def copy_state(self):
        return (self.tokens.copy(), self.mask.copy(), self.in_block.copy(),
                self.blk_meta.copy())


def window_sizes(shape: Shape) -> np.ndarray:
    if shape.windows is not None:
        w = np.asarray(shape.windows, dtype=np.int32)
        assert w.size == shape.batch
        return w
    lo, hi = shape.window_range
    u = uniform01(shape.seed, T_WIN, shape.batch)
    return (lo + np.floor(u * (hi - lo + 1))).astype(np.int32)


def _masks(shape: Shape, w: np.ndarray) -> np.ndarray:
    out = []
    for b, wb in enumerate(w):
        n_m = int(round(shape.mask_frac * int(wb)))
        u = uniform01(shape.seed, T_PERM + 1000 * (b + 1), int(wb))
        order = np.argsort(u, kind="stable")
        m = np.zeros(int(wb), dtype=np.uint8)
        m[order[:n_m]] = 1
        out.append(m)
    return np.concatenate(out) if out else np.zeros(0, np.uint8)


def make_step_inputs(shape: Shape, weights: bool = True,
                     prefix_lens: Optional[np.ndarray] = None) -> StepInputs:
    """Inputs of one selection step (no active block) for `shape`."""
    s = shape.seed
    B = shape.batch
    w = window_sizes(shape)
    cu = np.zeros(B + 1, dtype=np.int32)
    cu[1:] = np.cumsum(w)
    R = int(cu[-1])
    P = shape.prefix
    pl = (np.full(B, P, dtype=np.int32) if prefix_lens is None
          else np.asarray(prefix_lens, dtype=np.int32))
    row_pos = np.concatenate([pl[b] + np.arange(w[b], dtype=np.int32)
                              for b in range(B)]).astype(np.int32)
    d, Hq, Hkv, D = shape.d_model, shape.n_heads_q, shape.n_heads_kv, shape.head_dim

    z = normal_f32(s, T_HID, R * d).reshape(R, d)
    u = uniform01(s, T_HSCALE, R)
    lo, hi = math.log(shape.hid_scale_lo), math.log(shape.hid_scale_hi)
    scale = np.exp(lo + u * (hi - lo)).astype(np.float32)
    hidden = f32_to_bf16_bits(z * scale[:, None])

    q = normal_bf16(s, T_Q, (R, Hq, D))
    k_win = normal_bf16(s, T_KWIN, (R, Hkv, D))
    v_win = normal_bf16(s, T_VWIN, (R, Hkv, D))
    k_cache = normal_bf16(s, T_KC, (B, P, Hkv, D))
    v_cache = normal_bf16(s, T_VC, (B, P, Hkv, D))
    if weights:
        w_lm = _big_weight(s, T_WLM, shape.vocab, d, shape.w_lm_std)
        w_emb = _big_weight(s, T_WEMB, shape.vocab, shape.d_base, shape.w_emb_std)
    else:
        w_lm = np.zeros((0, d), np.uint16)
        w_emb = np.zeros((0, shape.d_base), np.uint16)

    mask = _masks(shape, w)
    ut = uniform01(s, T_TOK, R)
    tokens = np.floor(ut * shape.vocab).astype(np.int32)
    tokens[mask == 1] = MASK_TOKEN
    return StepInputs(shape=shape, cu_rows=cu, prefix_len=pl, row_pos=row_pos,
                      hidden=hidden, q=q, k_win=k_win, v_win=v_win,
                      k_cache=k_cache, v_cache=v_cache, w_lm=w_lm, w_emb=w_emb,
                      tokens=tokens, mask=mask,
                      in_block=np.zeros(R, np.uint8),
                      blk_meta=np.zeros((B, 2), np.int32))


def preset_in_block(inp: StepInputs, span: int = 20) -> StepInputs:
    """Turn `inp` into an in-block step: each sequence's first `span` window
    rows form the active block, selected earlier with size `span`."""
    in_block = np.zeros_like(inp.in_block)
    meta = np.zeros_like(inp.blk_meta)
    for b in range(inp.shape.batch):
        r0, r1 = int(inp.cu_rows[b]), int(inp.cu_rows[b + 1])
        n = min(span, r1 - r0)
        if n == 0 or inp.mask[r0:r0 + n].sum() == 0:
            continue
        in_block[r0:r0 + n] = 1
        meta[b] = (inp.row_pos[r0], n)
    inp.in_block = in_block
    inp.blk_meta = meta
    return inp


def _row(seed: int, tid: int, key: int, n: int) -> np.ndarray:
    """n standard normals keyed by (seed, tid, key); for small rows."""
    return _gen(seed, tid, key).standard_normal(n, dtype=np.float32)


def with_suffix_cache(inp: StepInputs, suffix: int):
    """A copy of `inp` whose K/V cache also holds the positions after each
    window: capacity prefix + max window + suffix, the new positions drawn
    N(0,1) like the prefix.  Returns (inputs, suffix ranges [B][2] =
    {first position after the window, suffix})."""
    sh = inp.shape
    B, P, Hkv, D = inp.k_cache.shape
    w = np.diff(inp.cu_rows).astype(np.int64)
    extra = int(w.max()) + suffix
    k_ext = normal_bf16(sh.seed, T_KSUF, (B, extra, Hkv, D))
    v_ext = normal_bf16(sh.seed, T_VSUF, (B, extra, Hkv, D))
    out = dataclasses.replace(inp, k_cache=np.concatenate([inp.k_cache, k_ext], axis=1),
                              v_cache=np.concatenate([inp.v_cache, v_ext], axis=1))
    rng = np.stack([inp.prefix_len.astype(np.int64) + w, np.full(B, suffix)], axis=1)
    return out, rng.astype(np.int32)


def loop_window_inputs(shape: Shape, step: int, positions: np.ndarray):
    """Per-step tensors of the generation loop for the window `positions`
    (absolute positions).  Hidden states and queries depend on
    (seed, step, position); keys/values depend on (seed, position) only, so a
    position's K/V is the same in the window and later in the prefix cache.
    The hidden scale drifts toward peaked as the loop advances:
    s(step, pos) = min(s_pos * exp(0.05 * step), 64)."""
    s = shape.seed
    d, Hq, Hkv, D = shape.d_model, shape.n_heads_q, shape.n_heads_kv, shape.head_dim
    R = positions.size
    hid = np.empty((R, d), np.float32)
    q = np.empty((R, Hq * D), np.float32)
    lo, hi = math.log(shape.hid_scale_lo), math.log(shape.hid_scale_hi)
    for j, pos in enumerate(positions.tolist()):
        key = ((step & 0xFFFF) << 16) | (pos & 0xFFFF)
        hid[j] = _row(s, T_LOOPHID, key, d)
        q[j] = _row(s, T_LOOPQ, key, Hq * D)
        u = _gen(s, T_HSCALE, 0x10000 | (pos & 0xFFFF)).random()
        sc = min(math.exp(lo + u * (hi - lo)) * math.exp(0.05 * step), 64.0)
        hid[j] *= np.float32(sc)
    k, v = loop_kv(shape, positions)
    return (f32_to_bf16_bits(hid), f32_to_bf16_bits(q).reshape(R, Hq, D), k, v)


def loop_kv(shape: Shape, positions: np.ndarray):
    """K/V rows of the loop workload at absolute `positions`."""
    s = shape.seed
    Hkv, D = shape.n_heads_kv, shape.head_dim
    R = positions.size
    k = np.empty((R, Hkv * D), np.float32)
    v = np.empty((R, Hkv * D), np.float32)
    for j, pos in enumerate(positions.tolist()):
        k[j] = _row(s, T_LOOPKV, 2 * pos, Hkv * D)
        v[j] = _row(s, T_LOOPKV, 2 * pos + 1, Hkv * D)
    return (f32_to_bf16_bits(k).reshape(R, Hkv, D),
            f32_to_bf16_bits(v).reshape(R, Hkv, D))
