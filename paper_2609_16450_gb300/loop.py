"""Host driver of the generation loop (App. E algorithm, in the block-forward
window setting of Sec. 6.4) for one sequence: a committed prompt of
`prefix` positions followed by `gen_len` masked response positions.

Each step asks the library for the next window (ebd_loop_window), has the
caller supply that window's backbone outputs (hidden states, q, k, v) and
runs ebd_step on it.  The decode state (tokens, mask, block flags, block
meta) of the whole response stays on the device; a step's window is a slice
of it.  The K/V cache is indexed by absolute position; a step attends to its
first prefix + frontier rows (prefix cache) and, with cache='dual', also to
the positions right of the window (dual cache, Sec. 6.3).  With append=True
each step writes the K/V of the rows it commits into the cache
(ebd_step_args.kv_append); the cache then starts with the prompt only.
This module only marshals buffers; the window rule and every step of the
method run in the library."""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Callable, List, Optional

import numpy as np
import torch

from . import _ebd as E
from . import runtime as rt

MASK_TOKEN = -1


@dataclass
class LoopStep:
    step: int
    window: tuple
    accepted: np.ndarray
    argmax: np.ndarray
    conf: np.ndarray
    lbs_logit: np.ndarray
    lps_prob: np.ndarray
    attn_out: Optional[np.ndarray]
    device_us: float
    # the window's statistics and decode state before and after the step
    entropy: Optional[np.ndarray] = None
    ent_norm: Optional[np.ndarray] = None
    gap: Optional[np.ndarray] = None
    before: Optional[dict] = None
    after: Optional[dict] = None


@dataclass
class LoopResult:
    tokens: np.ndarray
    steps: int
    commits: List[int] = field(default_factory=list)
    records: List[LoopStep] = field(default_factory=list)
    device_us: float = 0.0
    k_cache: Optional[np.ndarray] = None  # [P0 + L][Hkv][D] int16 bits after the loop
    v_cache: Optional[np.ndarray] = None


def config_for_loop(shape, max_window: int = 64, decode_mode: int = E.EBD_DECODE_EB,
                    top_m: int = 1) -> E.ebd_config:
    return rt.config_for(shape, max_batch=1, max_window=max_window, max_rows=max_window,
                         max_prefix=shape.prefix + shape.gen_len, decode_mode=decode_mode,
                         top_m=top_m)


def run_loop(h: rt.Handle, shape, weights: rt.DeviceWeights,
             window_inputs: Callable, kv_rows: Callable, attention: bool = True,
             max_steps: Optional[int] = None, max_window: int = 64,
             keep: bool = True, stream: Optional[torch.cuda.Stream] = None,
             block: int = 32, cache: str = "prefix", append: bool = False,
             window: str = "block") -> LoopResult:
    """window_inputs(step, positions) -> (hidden, q, k_win, v_win) as bf16 bit
    arrays; kv_rows(positions) -> (k, v).  Positions are absolute.  Under the
    handle's baseline decode modes the window is the active fixed block of
    `block` positions (ebd_loop_block_window).  cache: 'prefix' or 'dual';
    append: the step appends committed rows' K/V to the cache, which starts
    with the prompt's K/V only (with 'dual', with every position's, the
    positions right of the window standing for the K/V a dual cache holds)."""
    if cache not in ("prefix", "dual"):
        raise ValueError("cache must be 'prefix' or 'dual'")
    if window not in ("block", "full"):
        raise ValueError("window must be 'block' or 'full'")
    full = window == "full"  # the full-sequence setting: the window is the whole response
    if full and (attention or append):
        raise ValueError("the full-sequence window runs without the window attention")
    fixed = h.cfg.decode_mode != E.EBD_DECODE_EB
    dev = "cuda"
    P0, L = shape.prefix, shape.gen_len
    d, Hq, Hkv, D = shape.d_model, shape.n_heads_q, shape.n_heads_kv, shape.head_dim
    W = L if full else max_window
    stream = stream or torch.cuda.current_stream()
    sid = stream.cuda_stream
    i32 = dict(dtype=torch.int32, device=dev)
    u8 = dict(dtype=torch.uint8, device=dev)
    f32 = dict(dtype=torch.float32, device=dev)
    tokens = torch.full((L,), MASK_TOKEN, **i32)
    mask = torch.ones((L,), **u8)
    in_block = torch.zeros((L,), **u8)
    meta = torch.zeros((2,), **i32)
    mask_h = np.ones(L, np.uint8)
    ib_h = np.zeros(L, np.uint8)
    meta_h = np.zeros(2, np.int32)
    # window inputs, outputs and the K/V of every position
    hid = torch.empty((W, d), dtype=torch.int16, device=dev)
    q = torch.empty((W, Hq, D), dtype=torch.int16, device=dev)
    kw = torch.empty((W, Hkv, D), dtype=torch.int16, device=dev)
    vw = torch.empty((W, Hkv, D), dtype=torch.int16, device=dev)
    cu = torch.zeros((2,), **i32)
    pl = torch.zeros((1,), **i32)
    rp = torch.zeros((W,), **i32)
    outs = {k: torch.empty((W,), **f32) for k in ("conf", "entropy", "ent_norm", "gap",
                                                  "lbs_logit", "lps_prob")}
    argmax = torch.empty((W,), **i32)
    accepted = torch.empty((W,), **u8)
    attn_out = torch.empty((W, Hq, D), **f32) if attention else None
    kc = vc = None
    sfx = torch.zeros((2,), **i32)
    if attention or append:
        n0 = P0 if (append and cache == "prefix") else P0 + L
        kk, vv = kv_rows(np.arange(n0, dtype=np.int32))
        kc = torch.zeros((1, P0 + L, Hkv, D), dtype=torch.int16, device=dev)
        vc = torch.zeros((1, P0 + L, Hkv, D), dtype=torch.int16, device=dev)
        kc[0, :n0] = rt._dev(kk, dev).reshape(n0, Hkv, D)
        vc[0, :n0] = rt._dev(vv, dev).reshape(n0, Hkv, D)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    res = LoopResult(tokens=None, steps=0)
    step = 0
    while True:
        if max_steps is not None and step >= max_steps:
            break
        if full:
            s, lo, hi = E.EBD_OK, (0 if mask_h.any() else L), L
        elif fixed:
            s, lo, hi = E.ebd_loop_block_window(mask_h, block)
        else:
            s, lo, hi = E.ebd_loop_window(mask_h, ib_h, meta_h, W)
        if s != E.EBD_OK:
            raise E.EbdError(s, "loop window")
        if lo >= L:
            break
        R = hi - lo
        positions = (P0 + np.arange(lo, hi)).astype(np.int32)
        h_b, q_b, k_b, v_b = window_inputs(step, positions)
        with torch.cuda.stream(stream):
            hid[:R].copy_(torch.from_numpy(np.ascontiguousarray(h_b).view(np.int16)).reshape(R, d))
            q[:R].copy_(torch.from_numpy(np.ascontiguousarray(q_b).view(np.int16)).reshape(R, Hq, D))
            kw[:R].copy_(torch.from_numpy(np.ascontiguousarray(k_b).view(np.int16)).reshape(R, Hkv, D))
            vw[:R].copy_(torch.from_numpy(np.ascontiguousarray(v_b).view(np.int16)).reshape(R, Hkv, D))
            cu.copy_(torch.tensor([0, R], dtype=torch.int32))
            pl.copy_(torch.tensor([P0 + lo], dtype=torch.int32))
            rp[:R].copy_(torch.from_numpy(positions))
            sfx.copy_(torch.tensor([P0 + hi, L - hi], dtype=torch.int32))
        a = E.ebd_step_args()
        a.batch, a.rows = 1, R
        a.cu_rows, a.prefix_len, a.row_pos = cu.data_ptr(), pl.data_ptr(), rp.data_ptr()
        a.hidden, a.q, a.k_win, a.v_win = hid.data_ptr(), q.data_ptr(), kw.data_ptr(), vw.data_ptr()
        if attention or append:
            a.k_cache, a.v_cache = kc.data_ptr(), vc.data_ptr()
        if attention:
            a.attn_out = attn_out.data_ptr()
            if cache == "dual":
                a.suffix = sfx.data_ptr()
        a.kv_append = 1 if append else 0
        a.w_lm, a.w_lm_layout = weights.w_lm.data_ptr(), weights.layout
        a.tokens = tokens.data_ptr() + 4 * lo
        a.mask = mask.data_ptr() + lo
        a.in_block = in_block.data_ptr() + lo
        a.blk_meta = meta.data_ptr()
        for k, t in outs.items():
            setattr(a, k, t.data_ptr())
        a.argmax, a.accepted = argmax.data_ptr(), accepted.data_ptr()
        before = int(mask_h.sum())
        if keep:
            snap = dict(tokens=tokens[lo:hi].cpu().numpy(), mask=mask_h[lo:hi].copy(),
                        in_block=ib_h[lo:hi].copy(), meta=meta_h.copy())
        ev0.record(stream)
        E.check(E.ebd_step(h.h, a, sid), h.h)
        ev1.record(stream)
        st = h.sync_status(stream)
        if st != 0:
            raise E.EbdError(st, E.ebd_last_error(h.h))
        us = ev0.elapsed_time(ev1) * 1000.0
        mask_h = mask.cpu().numpy()
        ib_h = in_block.cpu().numpy()
        meta_h = meta.cpu().numpy()
        if keep:
            after = dict(tokens=tokens[lo:hi].cpu().numpy(), mask=mask_h[lo:hi].copy(),
                         in_block=ib_h[lo:hi].copy(), meta=meta_h.copy())
        if meta_h[1] == 0 and ib_h.any():
            # a resolved block releases its flags outside the window too
            in_block.zero_()
            ib_h[:] = 0
        res.commits.append(before - int(mask_h.sum()))
        res.device_us += us
        if keep:
            res.records.append(LoopStep(
                step=step, window=(lo, hi), accepted=accepted[:R].cpu().numpy(),
                argmax=argmax[:R].cpu().numpy(), conf=outs["conf"][:R].cpu().numpy(),
                lbs_logit=outs["lbs_logit"][:R].cpu().numpy(),
                lps_prob=outs["lps_prob"][:R].cpu().numpy(),
                attn_out=attn_out[:R].cpu().numpy() if attention else None, device_us=us,
                entropy=outs["entropy"][:R].cpu().numpy(), ent_norm=outs["ent_norm"][:R].cpu().numpy(),
                gap=outs["gap"][:R].cpu().numpy(), before=snap, after=after))
        step += 1
    res.tokens = tokens.cpu().numpy()
    res.steps = step
    if kc is not None:
        res.k_cache, res.v_cache = kc[0].cpu().numpy(), vc[0].cpu().numpy()
    return res
