"""Parameter list and seeded random init of the two routers.

Architectures (App. C.1 for LBS, App. D.1 for LPS):
  LBS  F_ent = Linear(1->64) -> GELU -> Linear(64->64) -> LayerNorm
       W_tok: Linear(d_base->64) on the frozen embedding W_e[x_hat]
       W_combine: Linear(128->128); E_pos: L x 128
       2 encoder layers (d=128, 4 heads, FFN 256, GELU); head Linear(128->1)
  LPS  Linear(5->32) -> LayerNorm -> GELU; 2 pre-norm blocks (d=32,
       4 heads, FFN 64, GELU); head Linear(32->1)

The blob order below is an interface (the C library documents and
reproduces it): every tensor row-major, bf16, concatenated in this order.

The paper gives no trained weights, so the routers are random-init in the
style of PyTorch defaults: Linear weight and bias ~ U(-1/sqrt(fan_in),
+1/sqrt(fan_in)), LayerNorm gain 1 and bias 0, and E_pos ~ U(-a, a) with
a = 0.02*sqrt(3) (std 0.02).  Uniforms come from SplitMix64 (Steele, Lea &
Flood, OOPSLA 2014) used as a counter-based generator:
  GAMMA = 0x9E3779B97F4A7C15
  mix(z): z = (z ^ z>>30) * 0xBF58476D1CE4E5B9
          z = (z ^ z>>27) * 0x94D049BB133111EB
          return z ^ z>>31
  key_t = mix(seed ^ ((t + 1) * GAMMA))          (t: tensor index)
  z_i   = mix(key_t + (i + 1) * GAMMA)            (i: element index)
  u_i   = (z_i >> 40) * 2^-24                     (float32, exact)
  w_i   = bf16_rne( float32(2*u_i - 1) * float32(bound) )
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import Dict, List, Tuple

import numpy as np

from .gen import bf16_to_f32, f32_to_bf16_bits

_GAMMA = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)
_MASK64 = (1 << 64) - 1


def _mix_np(z: np.ndarray) -> np.ndarray:
    with np.errstate(over="ignore"):
        z = (z ^ (z >> np.uint64(30))) * _M1
        z = (z ^ (z >> np.uint64(27))) * _M2
        return z ^ (z >> np.uint64(31))


def _mix_int(z: int) -> int:
    z &= _MASK64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _MASK64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _MASK64
    return z ^ (z >> 31)


def splitmix64_uniform(seed: int, t: int, n: int) -> np.ndarray:
    """u_i in [0,1) as float32 (24-bit) for tensor index t."""
    key = _mix_int((seed ^ (((t + 1) * 0x9E3779B97F4A7C15) & _MASK64)) & _MASK64)
    i = np.arange(1, n + 1, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = _mix_np(np.uint64(key) + i * _GAMMA)
    return (z >> np.uint64(40)).astype(np.float32) * np.float32(2.0 ** -24)


@dataclass(frozen=True)
class Tensor:
    name: str
    shape: Tuple[int, ...]
    init: str          # "lin", "ones", "zeros", "pos"
    fan_in: int = 0

    @property
    def size(self) -> int:
        return int(np.prod(self.shape))


@dataclass(frozen=True)
class RouterLayout:
    d_base: int
    gen_len: int
    tensors: Tuple[Tensor, ...]

    @property
    def offsets(self) -> Dict[str, Tuple[int, Tuple[int, ...]]]:
        off, out = 0, {}
        for t in self.tensors:
            out[t.name] = (off, t.shape)
            off += t.size
        return out

    @property
    def total(self) -> int:
        return sum(t.size for t in self.tensors)

    def count(self, prefix: str) -> int:
        return sum(t.size for t in self.tensors if t.name.startswith(prefix))


def router_layout(d_base: int, gen_len: int) -> RouterLayout:
    T: List[Tensor] = []

    def lin(name, n_out, n_in):
        T.append(Tensor(name + ".w", (n_out, n_in), "lin", n_in))
        T.append(Tensor(name + ".b", (n_out,), "lin", n_in))

    def ln(name, n):
        T.append(Tensor(name + ".g", (n,), "ones"))
        T.append(Tensor(name + ".b", (n,), "zeros"))

    # LBS router (App. C.1)
    lin("lbs.ent1", 64, 1)
    lin("lbs.ent2", 64, 64)
    ln("lbs.ent_ln", 64)
    lin("lbs.tok", 64, d_base)
    lin("lbs.comb", 128, 128)
    T.append(Tensor("lbs.pos", (gen_len, 128), "pos"))
    for l in range(2):
        p = f"lbs.l{l}"
        lin(p + ".qkv", 384, 128)
        lin(p + ".out", 128, 128)
        ln(p + ".ln1", 128)
        lin(p + ".ff1", 256, 128)
        lin(p + ".ff2", 128, 256)
        ln(p + ".ln2", 128)
    lin("lbs.head", 1, 128)
    # LPS router (App. D.1)
    lin("lps.in", 32, 5)
    ln("lps.in_ln", 32)
    for l in range(2):
        p = f"lps.l{l}"
        ln(p + ".ln1", 32)
        lin(p + ".qkv", 96, 32)
        lin(p + ".out", 32, 32)
        ln(p + ".ln2", 32)
        lin(p + ".ff1", 64, 32)
        lin(p + ".ff2", 32, 64)
    lin("lps.head", 1, 32)
    return RouterLayout(d_base=d_base, gen_len=gen_len, tensors=tuple(T))


def _init_tensor(seed: int, t_index: int, t: Tensor) -> np.ndarray:
    if t.init == "ones":
        return np.full(t.size, 0x3F80, dtype=np.uint16)
    if t.init == "zeros":
        return np.zeros(t.size, dtype=np.uint16)
    u = splitmix64_uniform(seed, t_index, t.size)
    v = np.float32(2.0) * u - np.float32(1.0)
    if t.init == "lin":
        bound = np.float32(1.0) / np.sqrt(np.float32(t.fan_in))
    elif t.init == "pos":
        bound = np.float32(0.02) * np.sqrt(np.float32(3.0))
    else:
        raise ValueError(t.init)
    return f32_to_bf16_bits((v * bound).astype(np.float32))


def router_weights(seed: int, d_base: int, gen_len: int) -> Dict[str, np.ndarray]:
    """Named bf16 tensors (uint16 bits) of both routers."""
    lay = router_layout(d_base, gen_len)
    return {t.name: _init_tensor(seed, i, t).reshape(t.shape)
            for i, t in enumerate(lay.tensors)}


def pack_blob(weights: Dict[str, np.ndarray], d_base: int, gen_len: int) -> np.ndarray:
    lay = router_layout(d_base, gen_len)
    return np.concatenate([np.asarray(weights[t.name], np.uint16).reshape(-1)
                           for t in lay.tensors])


def unpack_blob(blob: np.ndarray, d_base: int, gen_len: int) -> Dict[str, np.ndarray]:
    lay = router_layout(d_base, gen_len)
    out, off = {}, 0
    for t in lay.tensors:
        out[t.name] = np.asarray(blob[off:off + t.size], np.uint16).reshape(t.shape)
        off += t.size
    assert off == blob.size, (off, blob.size)
    return out


def weights_f64(weights: Dict[str, np.ndarray]) -> Dict[str, np.ndarray]:
    return {k: bf16_to_f32(v).astype(np.float64) for k, v in weights.items()}
