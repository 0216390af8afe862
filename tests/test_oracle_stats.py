"""Pins of the oracle's LM-head statistics (no GPU).

Each check ties the oracle to something other than itself: hand-worked values
(tests/golden/softmax_stats.json), closed forms (uniform, one-hot, k-way
ties), SciPy's softmax/entropy routines, exact rational arithmetic for the
LM-head dot products, and the shift invariance of softmax.
"""
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest
from scipy.special import softmax as sp_softmax
from scipy.stats import entropy as sp_entropy

from oracle import ebd_oracle as o

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def test_golden_hand_worked():
    g = json.load(open(os.path.join(GOLD, "softmax_stats.json")))
    for c in g["cases"]:
        st = o.softmax_stats(np.array([c["logits"]]))
        assert st.argmax[0] == c["argmax"], c["note"]
        for k in ("conf", "gap", "entropy", "ent_norm"):
            assert abs(getattr(st, k)[0] - c[k]) < 1e-12, (k, c["note"])


@pytest.mark.parametrize("V", [2, 7, 4096, 126464])
def test_uniform_closed_form(V):
    st = o.softmax_stats(np.full((1, V), -3.25))
    assert st.entropy[0] == pytest.approx(math.log(V), abs=1e-9)
    assert st.ent_norm[0] == pytest.approx(1.0, abs=1e-12)
    assert st.conf[0] == pytest.approx(1.0 / V, rel=1e-12)
    assert st.gap[0] == 0.0 and st.argmax[0] == 0 and st.near_tie[0]


@pytest.mark.parametrize("V,idx", [(16, 0), (4096, 4095), (4096, 1234)])
def test_one_hot_closed_form(V, idx):
    l = np.zeros((1, V)); l[0, idx] = 1000.0
    st = o.softmax_stats(l)
    assert st.entropy[0] == pytest.approx(0.0, abs=1e-12)
    assert st.conf[0] == pytest.approx(1.0, abs=1e-12)
    assert st.gap[0] == pytest.approx(1.0, abs=1e-12)
    assert st.argmax[0] == idx and not st.near_tie[0]


@pytest.mark.parametrize("k", [2, 3, 5])
def test_k_way_tie(k):
    V = 64
    l = np.full((1, V), -2000.0)
    tied = [9, 3, 40, 17, 22][:k]
    l[0, tied] = 1.5
    st = o.softmax_stats(l)
    assert st.entropy[0] == pytest.approx(math.log(k), abs=1e-12)
    assert st.conf[0] == pytest.approx(1.0 / k, abs=1e-12)
    assert st.gap[0] == pytest.approx(0.0, abs=1e-15)
    assert st.argmax[0] == min(tied)


def test_against_scipy_random():
    rng = np.random.default_rng(5)
    for scale in (0.1, 1.0, 8.0, 40.0):
        l = rng.standard_normal((6, 1000)) * scale
        st = o.softmax_stats(l)
        p = sp_softmax(l, axis=1)
        srt = np.sort(p, axis=1)
        np.testing.assert_allclose(st.conf, srt[:, -1], rtol=1e-12)
        np.testing.assert_allclose(st.gap, srt[:, -1] - srt[:, -2], atol=1e-15)
        np.testing.assert_allclose(st.entropy, sp_entropy(p, axis=1), rtol=1e-10, atol=1e-13)
        np.testing.assert_allclose(st.ent_norm, sp_entropy(p, axis=1) / math.log(1000), rtol=1e-10, atol=1e-13)
        np.testing.assert_array_equal(st.argmax, np.argmax(l, axis=1))


def test_shift_invariance_and_bounds():
    rng = np.random.default_rng(6)
    l = rng.standard_normal((4, 333)) * 3
    a, b = o.softmax_stats(l), o.softmax_stats(l + 77.5)
    for k in ("conf", "entropy", "gap"):
        np.testing.assert_allclose(getattr(a, k), getattr(b, k), atol=1e-12)
    assert np.all(a.entropy >= 0) and np.all(a.entropy <= math.log(333) + 1e-12)
    assert np.all((a.conf > 0) & (a.conf <= 1)) and np.all(a.gap >= 0)


def test_lm_logits_exact_rationals():
    """bf16 products and short sums are exact in float64: compare against
    exact rational arithmetic on the decoded values."""
    rng = np.random.default_rng(7)
    H = rng.integers(0, 1 << 16, size=(3, 16), dtype=np.uint16)
    W = rng.integers(0, 1 << 16, size=(40, 16), dtype=np.uint16)
    # keep finite, moderate exponents
    H = (H & 0x83FF) | 0x3C00
    W = (W & 0x83FF) | 0x3800
    out = o.lm_logits(H, W, chunk=7)
    hf, wf = o.bf16(H), o.bf16(W)
    for r in range(3):
        for v in range(40):
            exact = sum(Fraction(float(hf[r, k])) * Fraction(float(wf[v, k])) for k in range(16))
            assert out[r, v] == float(exact)


def test_bf16_decode():
    assert o.bf16(np.array([0x3F80, 0xBF80, 0x4049, 0x0000], np.uint16)).tolist() == \
        [1.0, -1.0, 3.140625, 0.0]


# ---------------------------------------------------------------- vocabulary ranges
def _split_points(V, k, rng):
    cuts = np.sort(rng.choice(np.arange(1, V), size=k - 1, replace=False))
    return [0] + cuts.tolist() + [V]


@pytest.mark.parametrize("k", [1, 2, 3, 7])
def test_range_states_merge_to_the_whole_row(k):
    """The statistics merged from the states of any partition of the
    vocabulary equal the statistics of the whole row (scipy's softmax and
    entropy), whatever the order of the ranges."""
    rng = np.random.default_rng(40 + k)
    V = 997
    L = rng.standard_normal((5, V)) * np.array([[0.5], [2], [8], [20], [1]])
    L[4, 10] = L[4, 900] = L[4].max() + 3.0       # a duplicated maximum across ranges
    pts = _split_points(V, k, rng)
    states = [o.range_state(L[:, a:b], a) for a, b in zip(pts[:-1], pts[1:])]
    for order in (states, states[::-1]):
        st = o.merge_range_states(order, V)
        p = sp_softmax(L, axis=1)
        np.testing.assert_allclose(st.conf, p.max(axis=1), rtol=1e-12)
        np.testing.assert_allclose(st.entropy, sp_entropy(p, axis=1), rtol=1e-10, atol=1e-12)
        srt = np.sort(p, axis=1)
        np.testing.assert_allclose(st.gap, srt[:, -1] - srt[:, -2], rtol=1e-10, atol=1e-15)
        assert st.argmax.tolist() == np.argmax(L, axis=1).tolist()
    assert st.argmax[4] == 10 and st.gap[4] == 0.0  # lowest index of the duplicated maximum


def test_range_state_of_one_range_is_the_row():
    rng = np.random.default_rng(5)
    L = rng.standard_normal((3, 50)) * 4
    st = o.merge_range_states([o.range_state(L, 0)], 50)
    ref = o.softmax_stats(L)
    for k in ("conf", "entropy", "ent_norm", "gap"):
        np.testing.assert_allclose(getattr(st, k), getattr(ref, k), rtol=1e-12, atol=1e-15)
    assert st.argmax.tolist() == ref.argmax.tolist()


def test_range_state_single_entry_ranges():
    """Ranges of one entry each: m = the logit, S = 1, T = 0, l2 = -inf."""
    L = np.array([[1.0, 4.0, 4.0, -2.0]])
    states = [o.range_state(L[:, j:j + 1], j) for j in range(4)]
    assert states[2].S[0] == 1.0 and states[2].T[0] == 0.0 and states[2].l2[0] == -np.inf
    st = o.merge_range_states(states, 4)
    assert st.argmax[0] == 1 and st.gap[0] == 0.0
    np.testing.assert_allclose(st.conf[0], math.exp(4) / (math.exp(1) + 2 * math.exp(4) + math.exp(-2)),
                               rtol=1e-14)
