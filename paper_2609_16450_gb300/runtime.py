"""PyTorch plumbing around the C ABI: device buffers, streams and the
marshalling of ebd_step_args.  No step of the method runs here; every
computation is a kernel of libebd.so."""
from __future__ import annotations

import warnings
from dataclasses import dataclass
from typing import Dict, Optional

import numpy as np
import torch

from . import _ebd as E


def config_for(shape, max_batch=None, max_window=None, max_rows=None, max_prefix=None,
               debug_flags=0, **over) -> E.ebd_config:
    """ebd_config for a synth.Shape (or any object with the same fields)."""
    windows = shape.windows if shape.windows is not None else (shape.window_range[1],) * shape.batch
    mw = max_window or max(max(windows), 1)
    mb = max_batch or shape.batch
    c = E.ebd_config(
        d_model=shape.d_model, vocab=shape.vocab, n_heads_q=shape.n_heads_q,
        n_heads_kv=shape.n_heads_kv, head_dim=shape.head_dim, d_base=shape.d_base,
        max_batch=mb, max_window=mw, max_rows=max_rows or max(mb * mw, 1),
        max_prefix=shape.prefix if max_prefix is None else max_prefix, gen_len=shape.gen_len,
        g_max=shape.g_max, l_min=shape.l_min, l_b=shape.l_b, eos_id=shape.eos_id,
        lps_enabled=shape.lps_enabled, tau=shape.tau, tau_psi=shape.tau_psi,
        seed=shape.seed, debug_flags=debug_flags)
    for k, v in over.items():
        setattr(c, k, v)
    return c


def _dev(a: np.ndarray, device) -> torch.Tensor:
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint16:
        a = a.view(np.int16)
    with warnings.catch_warnings():
        warnings.simplefilter("ignore", UserWarning)  # read-only arrays are only read
        return torch.from_numpy(a).to(device, non_blocking=False)


def ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    return None if t is None else t.data_ptr()


class Handle:
    """Owns one ebd_handle; binds the token embedding once."""

    def __init__(self, cfg: E.ebd_config, w_emb: Optional[torch.Tensor] = None, stream=None):
        E.load()
        s, h = E.ebd_create(cfg)
        if s != E.EBD_OK:
            raise E.EbdError(s, "ebd_create failed")
        self.h = h
        self.cfg = cfg
        self.w_emb = None
        if w_emb is not None:
            self.bind(w_emb, stream)

    def bind(self, w_emb: torch.Tensor, stream=None):
        self.w_emb = w_emb
        E.check(E.ebd_bind_embedding(self.h, w_emb.data_ptr(), stream_handle(stream)), self.h)

    def sync_status(self, stream=None) -> int:
        return E.ebd_sync_status(self.h, stream_handle(stream))

    def close(self):
        if self.h is not None:
            E.ebd_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def stream_handle(stream) -> int:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


@dataclass
class DeviceWeights:
    w_lm: torch.Tensor
    w_emb: torch.Tensor
    layout: int = 0          # 0: row-major W_lm; 1: tiled by ebd_pack_lm_head


def upload_weights(inp, device="cuda") -> DeviceWeights:
    return DeviceWeights(w_lm=_dev(inp.w_lm, device), w_emb=_dev(inp.w_emb, device))


def pack_weights(h: "Handle", w: DeviceWeights, stream=None) -> DeviceWeights:
    """Tiled copy of W_lm (one-time); the row-major copy is released."""
    n = E.ebd_lm_head_packed_bytes(h.cfg)
    packed = torch.empty(n // 2, dtype=torch.int16, device=w.w_lm.device)
    E.check(E.ebd_pack_lm_head(h.h, w.w_lm.data_ptr(), packed.data_ptr(), stream_handle(stream)),
            h.h)
    torch.cuda.synchronize()
    return DeviceWeights(w_lm=packed, w_emb=w.w_emb, layout=1)


class DeviceStep:
    """Device copies of one step's inputs/state plus output buffers."""

    def __init__(self, inp, weights: DeviceWeights, device="cuda", attention=True,
                 outputs=True):
        sh = inp.shape
        self.inp = inp
        self.device = device
        self.batch = sh.batch
        self.rows = inp.rows
        R, Hq, D = self.rows, sh.n_heads_q, sh.head_dim
        self.weights = weights
        self.cu_rows = _dev(inp.cu_rows.astype(np.int32), device)
        self.prefix_len = _dev(inp.prefix_len.astype(np.int32), device)
        self.row_pos = _dev(inp.row_pos.astype(np.int32), device)
        self.hidden = _dev(inp.hidden, device)
        self.q = _dev(inp.q, device)
        self.k_win = _dev(inp.k_win, device)
        self.v_win = _dev(inp.v_win, device)
        self.k_cache = _dev(inp.k_cache, device)
        self.v_cache = _dev(inp.v_cache, device)
        self.attention = attention
        f32 = dict(dtype=torch.float32, device=device)
        self.attn_out = torch.empty((max(R, 1), Hq, D), **f32) if attention else None
        if outputs:
            self.conf = torch.empty(max(R, 1), **f32)
            self.entropy = torch.empty(max(R, 1), **f32)
            self.ent_norm = torch.empty(max(R, 1), **f32)
            self.gap = torch.empty(max(R, 1), **f32)
            self.lbs_logit = torch.empty(max(R, 1), **f32)
            self.lps_prob = torch.empty(max(R, 1), **f32)
            self.argmax = torch.empty(max(R, 1), dtype=torch.int32, device=device)
            self.accepted = torch.empty(max(R, 1), dtype=torch.uint8, device=device)
        else:
            self.conf = self.entropy = self.ent_norm = self.gap = None
            self.lbs_logit = self.lps_prob = self.argmax = self.accepted = None
        self.reset_state(inp)

    def reset_state(self, inp=None):
        inp = inp or self.inp
        self.tokens = _dev(inp.tokens.astype(np.int32), self.device)
        self.mask = _dev(inp.mask.astype(np.uint8), self.device)
        self.in_block = _dev(inp.in_block.astype(np.uint8), self.device)
        self.blk_meta = _dev(inp.blk_meta.astype(np.int32), self.device)
        self.state0 = (self.tokens.clone(), self.mask.clone(), self.in_block.clone(),
                       self.blk_meta.clone())

    def restore_state(self):
        """Device-side copy of the pristine state (keeps pointers fixed)."""
        for dst, src in zip((self.tokens, self.mask, self.in_block, self.blk_meta), self.state0):
            dst.copy_(src, non_blocking=True)

    def args(self) -> E.ebd_step_args:
        a = E.ebd_step_args()
        a.batch, a.rows = self.batch, self.rows
        for name in ("cu_rows", "prefix_len", "row_pos", "hidden", "q", "k_win", "v_win",
                     "k_cache", "v_cache", "tokens", "mask", "in_block", "blk_meta",
                     "attn_out", "conf", "entropy", "ent_norm", "gap", "argmax",
                     "lbs_logit", "lps_prob", "accepted"):
            setattr(a, name, ptr(getattr(self, name)))
        a.w_lm = self.weights.w_lm.data_ptr()
        a.w_lm_layout = self.weights.layout
        return a

    def fetch(self) -> Dict[str, np.ndarray]:
        torch.cuda.synchronize()
        R = self.rows
        out = dict(tokens=self.tokens.cpu().numpy(), mask=self.mask.cpu().numpy(),
                   in_block=self.in_block.cpu().numpy(), blk_meta=self.blk_meta.cpu().numpy())
        for k in ("conf", "entropy", "ent_norm", "gap", "lbs_logit", "lps_prob", "argmax",
                  "accepted"):
            t = getattr(self, k)
            if t is not None:
                out[k] = t[:R].cpu().numpy()
        if self.attn_out is not None:
            out["attn_out"] = self.attn_out[:R].cpu().numpy()
        return out
