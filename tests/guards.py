"""Guard words around device buffers (GPU tests): every buffer a step writes
is allocated with GUARD bytes of a fixed pattern before and after it; after
the step the guards must be unchanged, so that a kernel writing past either
end of a buffer is caught."""
from __future__ import annotations

import numpy as np

GUARD = 256       # bytes on each side (keeps the interior 256-byte aligned)
PATTERN = 0xA5

OUT_F32 = ("conf", "entropy", "ent_norm", "gap", "lbs_logit", "lps_prob")


class Guarded:
    def __init__(self, torch, n, dtype, fill=None):
        esz = torch.tensor([], dtype=dtype).element_size()
        g = GUARD // esz
        self.whole = torch.empty(n + 2 * g, dtype=dtype, device="cuda")
        self.whole.view(torch.uint8).fill_(PATTERN)
        self.t = self.whole[g:g + n]
        if fill is not None:
            self.t.copy_(fill)

    def intact(self) -> bool:
        import torch
        b = self.whole.view(torch.uint8)
        return bool((b[:GUARD] == PATTERN).all().item() and (b[-GUARD:] == PATTERN).all().item())


def guarded_step(E, rt, h, inp, w, attention=True, append=False, call="step", rows=None):
    """One ebd_step (or one stage call: call = 'attention' | 'lm_stats') with
    every written buffer guarded.  The per-row buffers hold inp.rows rows;
    `rows` (default inp.rows) is the row count the library is told, so a
    smaller value makes the row offsets in inp.cu_rows overrun it while every
    access still stays inside the allocations.  Returns (status, outputs as
    numpy, guard records)."""
    import torch
    sh = inp.shape
    RA = inp.rows
    R = RA if rows is None else rows
    B = len(inp.cu_rows) - 1
    pad = lambda a, n: np.concatenate([a, np.zeros((n - len(a),) + a.shape[1:], a.dtype)]) if n > len(a) else a
    dev = rt._dev
    g = {}
    for k in OUT_F32:
        g[k] = Guarded(torch, RA, torch.float32)
    g["argmax"] = Guarded(torch, RA, torch.int32)
    g["accepted"] = Guarded(torch, RA, torch.uint8)
    g["tokens"] = Guarded(torch, RA, torch.int32, torch.from_numpy(pad(inp.tokens.astype(np.int32), RA)))
    g["mask"] = Guarded(torch, RA, torch.uint8, torch.from_numpy(pad(inp.mask.astype(np.uint8), RA)))
    g["in_block"] = Guarded(torch, RA, torch.uint8, torch.from_numpy(pad(inp.in_block.astype(np.uint8), RA)))
    g["blk_meta"] = Guarded(torch, 2 * B, torch.int32, torch.from_numpy(inp.blk_meta.astype(np.int32).reshape(-1)))
    if attention:
        g["attn_out"] = Guarded(torch, RA * sh.n_heads_q * sh.head_dim, torch.float32)
    kc = vc = None
    if append:
        n = inp.k_cache.size
        g["k_cache"] = Guarded(torch, n, torch.int16, torch.from_numpy(inp.k_cache.view(np.int16).reshape(-1)))
        g["v_cache"] = Guarded(torch, n, torch.int16, torch.from_numpy(inp.v_cache.view(np.int16).reshape(-1)))
    keep = [dev(inp.cu_rows.astype(np.int32), "cuda"), dev(inp.prefix_len.astype(np.int32), "cuda"),
            dev(pad(inp.row_pos.astype(np.int32), RA), "cuda"),
            dev(inp.hidden.reshape(RA, -1), "cuda"),
            dev(inp.q.reshape(RA, -1), "cuda"), dev(inp.k_win.reshape(RA, -1), "cuda"),
            dev(inp.v_win.reshape(RA, -1), "cuda")]
    a = E.ebd_step_args()
    a.batch, a.rows = B, R
    a.cu_rows, a.prefix_len, a.row_pos, a.hidden, a.q, a.k_win, a.v_win = (t.data_ptr() for t in keep)
    if append:
        a.k_cache, a.v_cache = g["k_cache"].t.data_ptr(), g["v_cache"].t.data_ptr()
        a.kv_append = 1
    else:
        kc, vc = dev(inp.k_cache, "cuda"), dev(inp.v_cache, "cuda")
        keep += [kc, vc]
        a.k_cache, a.v_cache = kc.data_ptr(), vc.data_ptr()
    a.w_lm, a.w_lm_layout = w.w_lm.data_ptr(), w.layout
    for k, v in g.items():
        if k not in ("k_cache", "v_cache"):
            setattr(a, k, v.t.data_ptr())
    if not attention:
        a.attn_out = None
    fn = {"step": E.ebd_step, "attention": E.ebd_attention, "lm_stats": E.ebd_lm_stats}[call]
    E.check(fn(h.h, a, rt.stream_handle(None)), h.h)
    status = h.sync_status()
    torch.cuda.synchronize()
    out = {k: v.t[:R].cpu().numpy() if k not in ("blk_meta", "k_cache", "v_cache", "attn_out")
           else v.t.cpu().numpy() for k, v in g.items()}
    return status, out, g
