"""The C-ABI library without a GPU: it builds, loads, exports every function
include/ebd.h declares, and its host-only functions agree with the oracle
and with the seeded generators.  No compute call reaches a device here."""
import ctypes
import os
import re

import numpy as np
import pytest

import synth
from oracle import ebd_oracle as o

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import build
    build.build()
    return E.load()


def _declared():
    src = open(os.path.join(ROOT, "include", "ebd.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(ebd_[a-z_0-9]+)\s*\(", src)))


def test_every_declared_function_is_exported(lib):
    from paper_2609_16450_gb300 import _ebd as E
    names = _declared()
    assert len(names) >= 20
    for n in names:
        assert hasattr(lib, n), n
    assert sorted(E.EXPORTS) == names


def test_version(lib):
    from paper_2609_16450_gb300 import _ebd as E
    assert "sm_103a" in E.ebd_version()


def test_router_init_host_matches_generator(lib):
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    sh = synth.tiny
    cfg = rt.config_for(sh)
    s, blob = E.ebd_router_init_host(cfg)
    assert s == E.EBD_OK
    ref = synth.pack_blob(synth.router_weights(sh.seed, sh.d_base, sh.gen_len), sh.d_base,
                          sh.gen_len)
    np.testing.assert_array_equal(blob, ref)
    assert E.ebd_weight_count(cfg) == ref.size


def test_weight_count_at_paper_sizes(lib):
    """LBS 613,761 + LPS 17,377 parameters at L = 512, d_base = 4096."""
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    cfg = rt.config_for(synth.llada)
    assert E.ebd_weight_count(cfg) == 613_761 + 17_377


def test_create_without_a_device_fails_cleanly(lib):
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    torch = pytest.importorskip("torch")
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    s, h = E.ebd_create(rt.config_for(synth.tiny))
    assert s != E.EBD_OK and not h.value


def test_unsupported_config_is_rejected(lib):
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    cfg = rt.config_for(synth.tiny, head_dim=96)
    s, h = E.ebd_create(cfg)
    assert s == E.EBD_ERR_UNSUPPORTED and not h.value


def test_noalloc_argument_checks_need_no_device(lib):
    from paper_2609_16450_gb300 import _ebd as E
    big = E.EBD_NOALLOC_MAX_ROWS + 1
    assert E.ebd_lm_stats_noalloc(16, 16, 0, big, 256, 4096, 0, 0, 0, 0, 0, 16, 0) == \
        E.EBD_ERR_UNSUPPORTED
    assert E.ebd_lm_stats_noalloc(16, 16, 0, 4, 256, 4096, 0, 0, 0, 0, 0, 0, 0) == \
        E.EBD_ERR_INVALID_ARG
    assert E.ebd_lm_stats_noalloc(16, 16, 2, 4, 256, 4096, 0, 0, 0, 0, 0, 16, 0) == \
        E.EBD_ERR_INVALID_ARG
    assert E.ebd_lm_stats_noalloc(16, 16, 0, 0, 256, 4096, 0, 0, 0, 0, 0, 16, 0) == E.EBD_OK


def test_loop_window_matches_oracle(lib):
    """ebd_loop_window against the oracle's window rule on random states."""
    from paper_2609_16450_gb300 import _ebd as E
    rng = np.random.default_rng(7)
    for trial in range(400):
        L = int(rng.integers(1, 200))
        mask = (rng.random(L) < rng.random()).astype(np.uint8)
        ib = np.zeros(L, np.uint8)
        meta = np.zeros(2, np.int32)
        if mask.any() and rng.random() < 0.5:
            f = int(np.argmax(mask))
            span = int(rng.integers(1, 64))
            idx = f + np.sort(rng.choice(np.arange(min(span, L - f)), size=min(span, L - f) // 2 + 1,
                                         replace=False))
            ib[idx] = 1
            meta[:] = (int(idx[0]), idx.size)
        s, lo, hi = E.ebd_loop_window(mask, ib, meta, 64)
        assert s == E.EBD_OK
        if not mask.any():
            assert lo == hi == L
            continue
        f = int(np.argmax(mask))
        blk = [i for i in range(L) if ib[i]]
        assert (lo, hi) == o.loop_window(f, L, meta, blk), (trial, lo, hi)
    # invalid arguments and states
    assert E.ebd_loop_window(np.ones(4), np.zeros(4), np.array([0, 3]), 64)[0] == E.EBD_ERR_STATE
    assert E.ebd_loop_window(np.ones(4), np.zeros(4), np.zeros(2), 0)[0] == E.EBD_ERR_INVALID_ARG


def test_loop_block_window_matches_oracle(lib):
    from paper_2609_16450_gb300 import _ebd as E
    rng = np.random.default_rng(11)
    for _ in range(300):
        L = int(rng.integers(0, 150))
        mask = (rng.random(L) < rng.random() * 0.3).astype(np.uint8)
        block = int(rng.integers(1, 40))
        s, lo, hi = E.ebd_loop_block_window(mask, block)
        assert s == E.EBD_OK
        assert (lo, hi) == o.fixed_block_window(mask, block)
    assert E.ebd_loop_block_window(np.ones(4, np.uint8), 0)[0] == E.EBD_ERR_INVALID_ARG


def test_decode_mode_validation(lib):
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    for over in (dict(decode_mode=3), dict(decode_mode=E.EBD_DECODE_TOPM, top_m=0)):
        s, h = E.ebd_create(rt.config_for(synth.tiny, **over))
        assert s == E.EBD_ERR_UNSUPPORTED and not h.value
