"""bench.py's work model on CPU: the algorithmic bytes and FLOPs that the
roofline fractions divide by."""
import importlib.util
import os

import numpy as np

import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench():
    spec = importlib.util.spec_from_file_location("bench_mod", os.path.join(ROOT, "bench.py"))
    m = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(m)
    return m


def test_llada_step_bytes_and_flops():
    b = _bench()
    sh = synth.llada
    wk = b.step_work(sh, 32, 24, 152, True)
    assert wk["lm_bytes"] == 126464 * 4096 * 2 + 32 * 4096 * 2 + 32 * 152 * 20
    assert wk["lm_flops"] == 2 * 32 * 4096 * 126464
    kv = (512 + 32) * 32 * 128 * 2 * 2
    assert wk["attn_bytes"] == kv + 32 * 32 * 128 * (2 + 4)
    assert wk["attn_flops"] == 4 * 32 * (512 + 32) * 32 * 128


def test_dual_cache_suffix_counts_its_keys():
    b = _bench()
    sh = synth.llada
    S = b.suffix_len(sh)
    assert S == 512 - 32
    base = b.step_work(sh, 32, 24, 152, True)
    dual = b.step_work(sh, 32, 24, 152, True, suffix=S)
    assert dual["attn_bytes"] - base["attn_bytes"] == S * 32 * 128 * 2 * 2
    assert dual["attn_flops"] - base["attn_flops"] == 4 * 32 * S * 32 * 128
    app = b.step_work(sh, 32, 24, 152, True, suffix=S, append=True)
    assert app["attn_bytes"] - dual["attn_bytes"] == 32 * 32 * 128 * 2 * 2 * 2


def test_full_sequence_has_no_window_attention():
    b = _bench()
    assert b.full_sequence(synth.llada_full) and b.full_sequence(synth.loop_full)
    assert not b.full_sequence(synth.llada) and not b.full_sequence(synth.dream)
    wk = b.step_work(synth.llada_full, 512, 384, 152, True)
    assert wk["attn_bytes"] == 0 and wk["attn_flops"] == 0
    assert wk["lm_flops"] == 2 * 512 * 4096 * 126464
    assert np.isclose(wk["lm_flops"] / 1897.5e12 * 1e6, 279.5, atol=0.5)  # tensor roofline, us


def test_lm_grid_rule():
    """The LM-head grid: LLaDA-8B's 1976 units on 152 SMs go to 142 CTAs of at
    most 14 units; few units take one CTA each; a split that would drop
    below 90 % of the SMs keeps every SM."""
    b = _bench()
    assert b.lm_grid(152, 1976) == 142
    assert b.lm_grid(152, 2376) == 140
    assert b.lm_grid(152, 64) == 64
    assert b.lm_grid(152, 200) == 152  # 2 per CTA -> 3 per CTA would need only 67 CTAs
    for units in (153, 1000, 1976, 2376, 5000):
        g = b.lm_grid(152, units)
        assert -(-units // g) <= -(-units // 152) + 1
