"""Workload shapes of the decoding step (synthetic stand-ins).

The paper measures LLaDA-8B-Instruct, Dream-v0-Instruct-7B and LLaDA-1.5 on
GSM8K, MATH500, HumanEval and MBPP at generation length 512, base block 32,
threshold 0.9 (Sec. 6.1 and App. F).  None of those weights or datasets are
available, so every tensor here is drawn from a seeded counter-based
generator with the backbone's shapes; the value distributions below are the
recipe for those stand-ins.

Hyper-parameters follow App. F: g_max = 5, L_min = 8 (LLaDA, Dream),
tau = 0.9, tau_psi = 0.89 (LLaDA) / 0.90 (Dream); the fallback block is the
base block size L_B = 32 (Sec. 5.1, App. E).
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace
from typing import Optional, Tuple


@dataclass(frozen=True)
class Shape:
    name: str
    batch: int
    d_model: int
    vocab: int
    n_heads_q: int
    n_heads_kv: int
    head_dim: int
    prefix: int                      # cached prefix length of every sequence
    windows: Optional[Tuple[int, ...]]  # window rows per sequence (None: drawn)
    mask_frac: float                 # fraction of window rows that are masked
    gen_len: int                     # L (LBS positional table length)
    w_lm_std: float                  # std of the LM-head weights
    w_emb_std: float = 1.0           # std of the frozen token embedding
    window_range: Tuple[int, int] = (16, 64)  # when windows is None
    tau: float = 0.9
    tau_psi: float = 0.89
    l_min: int = 8
    g_max: int = 5
    l_b: int = 32
    lps_enabled: int = 1
    seed: int = 0
    hid_scale_lo: float = 0.5        # per-row hidden scale ~ logUniform[lo, hi]
    hid_scale_hi: float = 8.0

    @property
    def d_base(self) -> int:
        return self.d_model

    @property
    def eos_id(self) -> int:
        return self.vocab - 1

    def with_(self, **kw) -> "Shape":
        return replace(self, **kw)


# Tiny step: one small step the oracle finishes in seconds.
tiny = Shape(name="tiny", batch=1, d_model=256, vocab=4096, n_heads_q=4,
             n_heads_kv=4, head_dim=64, prefix=128, windows=(32,),
             mask_frac=0.75, gen_len=512, w_lm_std=0.02, seed=0)

# LLaDA-8B shaped step (hidden 4096, vocab 126464, 32x128 MHA).
llada = Shape(name="llada8b", batch=1, d_model=4096, vocab=126464,
              n_heads_q=32, n_heads_kv=32, head_dim=128, prefix=512,
              windows=(32,), mask_frac=0.75, gen_len=512,
              w_lm_std=1.0 / 64.0, seed=1)

# Dream-7B shaped step (hidden 3584, vocab 152064, GQA 28/4).
dream = Shape(name="dream7b", batch=8, d_model=3584, vocab=152064,
              n_heads_q=28, n_heads_kv=4, head_dim=128, prefix=1024,
              windows=None, mask_frac=0.75, gen_len=512,
              w_lm_std=1.0 / 64.0, tau_psi=0.90, seed=2)

# The full decoding loop at LLaDA-8B shape, prompt 256, gen 256.
loop_shape = Shape(name="loop_llada8b", batch=1, d_model=4096, vocab=126464,
                   n_heads_q=32, n_heads_kv=32, head_dim=128, prefix=256,
                   windows=(64,), mask_frac=1.0, gen_len=256,
                   w_lm_std=1.0 / 64.0, seed=3)

# the generation loop at the tiny shape: prompt 64, gen 64 (the oracle runs the
# whole loop in seconds)
loop_tiny = Shape(name="loop_tiny", batch=1, d_model=256, vocab=4096, n_heads_q=4,
                  n_heads_kv=4, head_dim=64, prefix=64, windows=(64,), mask_frac=1.0,
                  gen_len=64, w_lm_std=0.02, seed=4)

# The full-sequence setting (every position of the response is a row of the
# step; the LBS sees all masked positions; no KV cache): LLaDA-8B shapes with
# a 512-token response, and a tiny one the oracle finishes in seconds.
llada_full = Shape(name="llada8b_full", batch=1, d_model=4096, vocab=126464,
                   n_heads_q=32, n_heads_kv=32, head_dim=128, prefix=0,
                   windows=(512,), mask_frac=0.75, gen_len=512,
                   w_lm_std=1.0 / 64.0, seed=5)
tiny_full = Shape(name="tiny_full", batch=3, d_model=256, vocab=4096, n_heads_q=4,
                  n_heads_kv=4, head_dim=64, prefix=0, windows=(256, 100, 40),
                  mask_frac=0.75, gen_len=256, w_lm_std=0.02, seed=6)
# the generation loop in the full-sequence setting at the tiny shape (gen 96)
loop_full_tiny = Shape(name="loop_full_tiny", batch=1, d_model=256, vocab=4096, n_heads_q=4,
                       n_heads_kv=4, head_dim=64, prefix=64, windows=(96,), mask_frac=1.0,
                       gen_len=96, w_lm_std=0.02, seed=23)
# ... and at the LLaDA-8B loop shape (prompt 256, gen 256)
loop_full = loop_shape.with_(name="loop_full_llada8b", windows=(256,), seed=8)

SHAPES = {s.name: s for s in (tiny, llada, dream, loop_shape, loop_tiny, llada_full, tiny_full,
                              loop_full_tiny, loop_full)}


def sweep_points():
    """Throughput sweep: batch x cached prefix x window at the LLaDA-8B head shape."""
    pts = []
    k = 0
    for b in (1, 4, 16, 64):
        for p in (256, 1024, 4096):
            for w in (8, 32, 64):
                pts.append(llada.with_(name=f"sweep_b{b}_p{p}_w{w}", batch=b,
                                       prefix=p, windows=(w,) * b,
                                       mask_frac=0.6, seed=100 + k))
                k += 1
    return pts


def sweep_point(batch: int, prefix: int, window: int) -> Shape:
    for s in sweep_points():
        if s.batch == batch and s.prefix == prefix and s.windows[0] == window:
            return s
    raise KeyError((batch, prefix, window))
