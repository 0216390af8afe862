"""ctypes binding of libebd.so: the C functions of include/ebd.h under the
same names, with argument marshalling only.  Every function returns the C
status code (0 = EBD_OK) unless noted; `check()` turns a status into an
exception."""
from __future__ import annotations

import ctypes
import os
from ctypes import (POINTER, Structure, c_char_p, c_float, c_int32, c_size_t, c_uint64,
                    c_void_p)

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "libebd.so")

EBD_OK = 0
EBD_ERR_INVALID_ARG = -1
EBD_ERR_UNSUPPORTED = -2
EBD_ERR_CUDA = -3
EBD_ERR_TIMEOUT = -4
EBD_ERR_NONFINITE = -5
EBD_ERR_STATE = -6
EBD_ERR_BOUNDS = -7
EBD_DEBUG_FORCE_TIMEOUT = 1
EBD_DEBUG_FORCE_COPY_TIMEOUT = 2
EBD_DECODE_EB = 0
EBD_DECODE_THRESHOLD = 1
EBD_DECODE_TOPM = 2

STATUS_NAMES = {0: "EBD_OK", -1: "EBD_ERR_INVALID_ARG", -2: "EBD_ERR_UNSUPPORTED",
                -3: "EBD_ERR_CUDA", -4: "EBD_ERR_TIMEOUT", -5: "EBD_ERR_NONFINITE",
                -6: "EBD_ERR_STATE", -7: "EBD_ERR_BOUNDS"}


class ebd_config(Structure):
    _fields_ = [("d_model", c_int32), ("vocab", c_int32), ("n_heads_q", c_int32),
                ("n_heads_kv", c_int32), ("head_dim", c_int32), ("d_base", c_int32),
                ("max_batch", c_int32), ("max_window", c_int32), ("max_rows", c_int32),
                ("max_prefix", c_int32), ("gen_len", c_int32), ("g_max", c_int32),
                ("l_min", c_int32), ("l_b", c_int32), ("eos_id", c_int32),
                ("lps_enabled", c_int32), ("tau", c_float), ("tau_psi", c_float),
                ("seed", c_uint64), ("debug_flags", c_int32), ("decode_mode", c_int32),
                ("top_m", c_int32), ("reserved", c_int32)]


class ebd_step_args(Structure):
    _fields_ = [("batch", c_int32), ("rows", c_int32),
                ("cu_rows", c_void_p), ("prefix_len", c_void_p), ("row_pos", c_void_p),
                ("hidden", c_void_p), ("q", c_void_p), ("k_win", c_void_p), ("v_win", c_void_p),
                ("k_cache", c_void_p), ("v_cache", c_void_p), ("w_lm", c_void_p),
                ("tokens", c_void_p), ("mask", c_void_p), ("in_block", c_void_p),
                ("blk_meta", c_void_p), ("attn_out", c_void_p), ("conf", c_void_p),
                ("entropy", c_void_p), ("ent_norm", c_void_p), ("gap", c_void_p),
                ("argmax", c_void_p), ("lbs_logit", c_void_p), ("lps_prob", c_void_p),
                ("accepted", c_void_p), ("w_lm_layout", c_int32), ("kv_append", c_int32),
                ("suffix", c_void_p)]


EXPORTS = ["ebd_create", "ebd_destroy", "ebd_bind_embedding", "ebd_step", "ebd_step_host",
           "ebd_decide", "ebd_lm_stats", "ebd_attention", "ebd_sync_status",
           "ebd_export_weights", "ebd_import_weights", "ebd_router_init_host",
           "ebd_weight_count", "ebd_lm_head_packed_bytes", "ebd_pack_lm_head",
           "ebd_profile_enable", "ebd_profile_read", "ebd_last_error",
           "ebd_version", "ebd_lm_stats_noalloc", "ebd_loop_window",
           "ebd_loop_block_window", "ebd_lm_shard_state", "ebd_merge_shard_states"]

_lib = None


class EbdError(RuntimeError):
    def __init__(self, status, msg=""):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


def load(path: str = LIB_PATH):
    """Loads libebd.so (or the library named by the EBD_LIBRARY environment
    variable, e.g. the checked build); raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    path = os.environ.get("EBD_LIBRARY", path)
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with paper_2609_16450_gb300.build.build()")
    lib = ctypes.CDLL(path)
    P = POINTER
    lib.ebd_create.argtypes = [P(ebd_config), P(c_void_p)]
    lib.ebd_destroy.argtypes = [c_void_p]
    lib.ebd_destroy.restype = None
    lib.ebd_bind_embedding.argtypes = [c_void_p, c_void_p, c_void_p]
    for fn in ("ebd_step", "ebd_step_host", "ebd_decide", "ebd_lm_stats", "ebd_attention"):
        getattr(lib, fn).argtypes = [c_void_p, P(ebd_step_args), c_void_p]
    lib.ebd_sync_status.argtypes = [c_void_p, c_void_p]
    lib.ebd_export_weights.argtypes = [c_void_p, c_void_p, P(c_size_t)]
    lib.ebd_import_weights.argtypes = [c_void_p, c_void_p, c_size_t]
    lib.ebd_router_init_host.argtypes = [P(ebd_config), c_void_p, P(c_size_t)]
    lib.ebd_weight_count.argtypes = [P(ebd_config)]
    lib.ebd_weight_count.restype = c_size_t
    lib.ebd_last_error.argtypes = [c_void_p]
    lib.ebd_last_error.restype = c_char_p
    lib.ebd_lm_head_packed_bytes.argtypes = [P(ebd_config)]
    lib.ebd_lm_head_packed_bytes.restype = c_size_t
    lib.ebd_pack_lm_head.argtypes = [c_void_p, c_void_p, c_void_p, c_void_p]
    lib.ebd_profile_enable.argtypes = [c_void_p, c_int32]
    lib.ebd_profile_read.argtypes = [c_void_p, P(c_float)]
    lib.ebd_version.argtypes = []
    lib.ebd_lm_stats_noalloc.argtypes = [c_void_p, c_void_p, c_int32, c_int32, c_int32, c_int32,
                                         c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                                         c_void_p, c_void_p]
    lib.ebd_lm_stats_noalloc.restype = c_int32
    lib.ebd_loop_window.argtypes = [c_void_p, c_void_p, c_void_p, c_int32, c_int32, P(c_int32),
                                    P(c_int32)]
    lib.ebd_loop_window.restype = c_int32
    lib.ebd_loop_block_window.argtypes = [c_void_p, c_int32, c_int32, P(c_int32), P(c_int32)]
    lib.ebd_loop_block_window.restype = c_int32
    lib.ebd_lm_shard_state.argtypes = [c_void_p, P(ebd_step_args), c_int32, c_int32, c_void_p,
                                       c_void_p]
    lib.ebd_merge_shard_states.argtypes = [c_void_p, c_void_p, c_int32, P(ebd_step_args), c_void_p]
    lib.ebd_version.restype = c_char_p
    for fn in EXPORTS:
        if getattr(lib, fn).restype is ctypes.c_int:
            getattr(lib, fn).restype = c_int32
    _lib = lib
    return lib


def check(status: int, handle=None):
    if status != EBD_OK:
        msg = ebd_last_error(handle) if handle else ""
        raise EbdError(status, msg)


def ebd_create(cfg: ebd_config):
    """Returns (status, handle)."""
    h = c_void_p()
    s = load().ebd_create(ctypes.byref(cfg), ctypes.byref(h))
    return s, h


def ebd_destroy(h) -> None:
    load().ebd_destroy(h)


def ebd_bind_embedding(h, w_emb_ptr: int, stream: int = 0) -> int:
    return load().ebd_bind_embedding(h, c_void_p(w_emb_ptr), c_void_p(stream))


def ebd_step(h, args: ebd_step_args, stream: int = 0) -> int:
    return load().ebd_step(h, ctypes.byref(args), c_void_p(stream))


def ebd_step_host(h, args: ebd_step_args, stream: int = 0) -> int:
    return load().ebd_step_host(h, ctypes.byref(args), c_void_p(stream))


def ebd_decide(h, args: ebd_step_args, stream: int = 0) -> int:
    return load().ebd_decide(h, ctypes.byref(args), c_void_p(stream))


def ebd_lm_stats(h, args: ebd_step_args, stream: int = 0) -> int:
    return load().ebd_lm_stats(h, ctypes.byref(args), c_void_p(stream))


def ebd_lm_shard_state(h, args: ebd_step_args, v_off: int, v_count: int, state_ptr: int,
                       stream: int = 0) -> int:
    return load().ebd_lm_shard_state(h, ctypes.byref(args), v_off, v_count, c_void_p(state_ptr),
                                     c_void_p(stream))


def ebd_merge_shard_states(h, states_ptr: int, shards: int, args: ebd_step_args,
                           stream: int = 0) -> int:
    return load().ebd_merge_shard_states(h, c_void_p(states_ptr), shards, ctypes.byref(args),
                                         c_void_p(stream))


def ebd_attention(h, args: ebd_step_args, stream: int = 0) -> int:
    return load().ebd_attention(h, ctypes.byref(args), c_void_p(stream))


def ebd_sync_status(h, stream: int = 0) -> int:
    return load().ebd_sync_status(h, c_void_p(stream))


def ebd_export_weights(h):
    """Returns (status, bytes)."""
    import numpy as np
    n = c_size_t(0)
    s = load().ebd_export_weights(h, None, ctypes.byref(n))
    if s != EBD_OK:
        return s, None
    buf = np.empty(n.value // 2, dtype=np.uint16)
    s = load().ebd_export_weights(h, c_void_p(buf.ctypes.data), ctypes.byref(n))
    return s, buf


def ebd_import_weights(h, blob) -> int:
    import numpy as np
    blob = np.ascontiguousarray(blob, dtype=np.uint16)
    return load().ebd_import_weights(h, c_void_p(blob.ctypes.data), blob.nbytes)


def ebd_router_init_host(cfg: ebd_config):
    """Returns (status, uint16 blob)."""
    import numpy as np
    n = c_size_t(0)
    s = load().ebd_router_init_host(ctypes.byref(cfg), None, ctypes.byref(n))
    if s != EBD_OK:
        return s, None
    buf = np.empty(n.value // 2, dtype=np.uint16)
    s = load().ebd_router_init_host(ctypes.byref(cfg), c_void_p(buf.ctypes.data), ctypes.byref(n))
    return s, buf


def ebd_weight_count(cfg: ebd_config) -> int:
    return int(load().ebd_weight_count(ctypes.byref(cfg)))


def ebd_lm_head_packed_bytes(cfg: ebd_config) -> int:
    return int(load().ebd_lm_head_packed_bytes(ctypes.byref(cfg)))


def ebd_pack_lm_head(h, w_lm_ptr: int, w_packed_ptr: int, stream: int = 0) -> int:
    return load().ebd_pack_lm_head(h, c_void_p(w_lm_ptr), c_void_p(w_packed_ptr), c_void_p(stream))


def ebd_profile_enable(h, mode: int) -> int:
    """mode 0 off, 1 every kernel timed on its own, 2 production overlap."""
    return load().ebd_profile_enable(h, int(mode))


def ebd_profile_read(h):
    """Returns (status, [attention_ms, lm_head_ms, decision_ms])."""
    ms = (c_float * 3)()
    s = load().ebd_profile_read(h, ms)
    return s, [float(x) for x in ms]


def ebd_last_error(h) -> str:
    r = load().ebd_last_error(h)
    return r.decode() if r else ""


def ebd_version() -> str:
    return load().ebd_version().decode()


EBD_NOALLOC_MAX_ROWS = 64
EBD_NOALLOC_MAX_PARTS = 160


def ebd_lm_stats_noalloc(hidden_ptr: int, w_lm_ptr: int, w_lm_layout: int, rows: int,
                         d_model: int, vocab: int, conf_ptr: int, entropy_ptr: int,
                         ent_norm_ptr: int, gap_ptr: int, argmax_ptr: int, status_ptr: int,
                         stream: int = 0) -> int:
    """Allocation-free LM-head statistics; pointers are device addresses
    (0 for an output that is not wanted)."""
    return load().ebd_lm_stats_noalloc(hidden_ptr, w_lm_ptr, w_lm_layout, rows, d_model, vocab,
                                       conf_ptr or None, entropy_ptr or None, ent_norm_ptr or None,
                                       gap_ptr or None, argmax_ptr or None, status_ptr or None,
                                       stream or None)


def ebd_loop_window(mask, in_block, meta, max_window: int = 64):
    """mask, in_block: host uint8 [L]; meta: host int32 [2].  Returns
    (status, lo, hi)."""
    import numpy as np
    m = np.ascontiguousarray(mask, dtype=np.uint8)
    ib = np.ascontiguousarray(in_block, dtype=np.uint8)
    mt = np.ascontiguousarray(meta, dtype=np.int32)
    lo, hi = c_int32(0), c_int32(0)
    s = load().ebd_loop_window(m.ctypes.data, ib.ctypes.data, mt.ctypes.data, int(m.size),
                               int(max_window), ctypes.byref(lo), ctypes.byref(hi))
    return s, lo.value, hi.value


def ebd_loop_block_window(mask, block: int):
    """mask: host uint8 [L].  Returns (status, lo, hi)."""
    import numpy as np
    m = np.ascontiguousarray(mask, dtype=np.uint8)
    lo, hi = c_int32(0), c_int32(0)
    s = load().ebd_loop_block_window(m.ctypes.data, int(m.size), int(block), ctypes.byref(lo),
                                     ctypes.byref(hi))
    return s, lo.value, hi.value
