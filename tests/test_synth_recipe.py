"""The synthetic inputs follow their stated recipe (CPU, no GPU): shapes,
thresholds, masked fractions, window lengths, value distributions and
determinism of the seeded generators, for the configs the benchmark and the
GPU parity tests use."""
import numpy as np
import pytest

import synth


def _inp(sh, **kw):
    return synth.make_step_inputs(sh, weights=False, **kw)


@pytest.mark.parametrize("name,B,R,masked,P,V,tau_psi", [
    ("tiny", 1, 32, 24, 128, 4096, 0.89),
    ("llada", 1, 32, 24, 512, 126464, 0.89),
])
def test_single_window_configs(name, B, R, masked, P, V, tau_psi):
    sh = getattr(synth, name)
    inp = _inp(sh)
    assert sh.batch == B and inp.rows == R and int(inp.mask.sum()) == masked
    assert inp.prefix_len.tolist() == [P] and sh.vocab == V
    assert (sh.tau, sh.tau_psi, sh.l_min, sh.l_b, sh.g_max) == (0.9, tau_psi, 8, 32, 5)
    assert sh.eos_id == V - 1
    # masked rows carry no token; committed rows a vocabulary id
    assert np.all(inp.tokens[inp.mask == 1] == -1)
    assert np.all((inp.tokens[inp.mask == 0] >= 0) & (inp.tokens[inp.mask == 0] < V))


def test_dream_windows_and_mask_fraction():
    sh = synth.dream
    inp = _inp(sh)
    w = np.diff(inp.cu_rows)
    assert sh.batch == 8 and (w >= 16).all() and (w <= 64).all() and int(w.sum()) == inp.rows == 390
    assert (sh.n_heads_q, sh.n_heads_kv, sh.head_dim, sh.d_model, sh.vocab) == (28, 4, 128, 3584, 152064)
    assert inp.prefix_len.tolist() == [1024] * 8 and sh.tau_psi == 0.9
    for b in range(8):  # round(0.75 w_b) masked rows per sequence
        m = int(inp.mask[inp.cu_rows[b]:inp.cu_rows[b + 1]].sum())
        assert m == round(0.75 * w[b])


def test_sweep_grid():
    pts = synth.sweep_points()
    assert len(pts) == 36
    grid = {(s.batch, s.prefix, s.windows[0]) for s in pts}
    assert grid == {(b, p, w) for b in (1, 4, 16, 64) for p in (256, 1024, 4096) for w in (8, 32, 64)}
    assert len({s.seed for s in pts}) == 36 and all(s.mask_frac == 0.6 for s in pts)
    assert all(s.vocab == 126464 and s.d_model == 4096 and s.n_heads_q == s.n_heads_kv == 32 for s in pts)


def test_hidden_scale_and_bf16_values():
    """Hidden rows N(0,1) scaled per row by a log-uniform factor in [0.5, 8];
    every tensor holds bf16 bit patterns."""
    inp = synth.make_step_inputs(synth.tiny)
    h = synth.bf16_to_f32(inp.hidden).astype(np.float64)
    rms = np.sqrt((h ** 2).mean(axis=1))
    assert rms.min() > 0.5 * 0.8 and rms.max() < 8 * 1.2
    assert np.log(rms).max() - np.log(rms).min() > 1.0          # spread over the range
    for t in (inp.hidden, inp.q, inp.k_win, inp.v_win, inp.k_cache):
        assert t.dtype == np.uint16


def test_seeded_and_deterministic():
    a, b = _inp(synth.llada), _inp(synth.llada)
    for k in ("hidden", "q", "k_win", "v_win", "k_cache", "mask", "tokens", "row_pos"):
        assert np.array_equal(getattr(a, k), getattr(b, k)), k
    c = _inp(synth.llada.with_(seed=synth.llada.seed + 1))
    assert not np.array_equal(a.hidden, c.hidden)
