"""The oracle's pins are sensitive: each test here plants one plausible
mistake in the oracle (in this process only, through monkeypatch, on the CPU)
and checks that at least one of the pins that guard that part fails.

Mistakes planted: entropy in bits instead of nats; argmax ties to the highest
index; the gap against the third logit; an attention scale of 2/sqrt(D); one
prefix key dropped; GQA heads mapped round-robin instead of in groups; the
MaxGapFilter cut at a gap equal to g_max; the min-tokens fallback of L_min
rows instead of L_B; a strict kappa > tau in the accept rule; the tanh
approximation of GELU; a LayerNorm eps of 1e-6; an attention scale of
1/sqrt(d) instead of 1/sqrt(d/heads) in the routers; EOS kept among the
router candidates; the dual-cache suffix read one position late; the cache
append writing masked rows too; the LPS features in another order, pos
divided by |B n M|, rho over the whole window, GELU before LayerNorm in the
LPS input layer; in the LBS input (Eq. lbs_feat) the token branch first in
the fusion, E_pos added before W_combine, LayerNorm and GELU swapped in
F_ent."""
import numpy as np
import pytest

from oracle import ebd_oracle as o
from tests import test_oracle_attention as ta
from tests import test_oracle_decision as td
from tests import test_oracle_routers as tr
from tests import test_oracle_stats as ts


def _some_pin_fails(pins):
    """True if calling any of the pin callables raises AssertionError."""
    for pin in pins:
        try:
            pin()
        except AssertionError:
            return True
    return False


def _stats_pins():
    return [ts.test_golden_hand_worked,
            lambda: ts.test_uniform_closed_form(7),
            lambda: ts.test_one_hot_closed_form(16, 0),
            lambda: ts.test_k_way_tie(3),
            ts.test_against_scipy_random]


def test_the_pins_pass_as_they_stand():
    assert not _some_pin_fails(_stats_pins())
    assert not _some_pin_fails([ta.test_matches_torch_sdpa, ta.test_ragged_prefix_and_batch_separation,
                                ta.test_gqa_head_mapping])
    assert not _some_pin_fails([td.test_maxgap_golden, td.test_select_golden, td.test_accept_golden])


def test_entropy_in_bits_is_caught(monkeypatch):
    real = o.softmax_stats

    def bits(logits):
        st = real(logits)
        return o.RowStats(conf=st.conf, entropy=st.entropy / np.log(2.0), ent_norm=st.ent_norm, gap=st.gap,
                          argmax=st.argmax, logit_gap=st.logit_gap, near_tie=st.near_tie)
    monkeypatch.setattr(o, "softmax_stats", bits)
    assert _some_pin_fails(_stats_pins())


def test_argmax_ties_to_highest_index_are_caught(monkeypatch):
    real = o.softmax_stats

    def last(logits):
        st = real(logits)
        l = np.asarray(logits, np.float64)
        am = l.shape[1] - 1 - np.argmax(l[:, ::-1], axis=1)
        return o.RowStats(conf=st.conf, entropy=st.entropy, ent_norm=st.ent_norm, gap=st.gap,
                          argmax=am.astype(np.int64), logit_gap=st.logit_gap, near_tie=st.near_tie)
    monkeypatch.setattr(o, "softmax_stats", last)
    assert _some_pin_fails(_stats_pins())


def test_gap_against_the_third_logit_is_caught(monkeypatch):
    real = o.softmax_stats

    def third(logits):
        st = real(logits)
        l = np.sort(np.asarray(logits, np.float64), axis=1)[:, ::-1]
        m = l[:, 0:1]
        p = np.exp(l - m) / np.exp(l - m).sum(axis=1, keepdims=True)
        gap = p[:, 0] - (p[:, 2] if l.shape[1] > 2 else 0.0)
        return o.RowStats(conf=st.conf, entropy=st.entropy, ent_norm=st.ent_norm, gap=gap,
                          argmax=st.argmax, logit_gap=st.logit_gap, near_tie=st.near_tie)
    monkeypatch.setattr(o, "softmax_stats", third)
    assert _some_pin_fails(_stats_pins())


def test_wrong_attention_scale_is_caught(monkeypatch):
    """scale 2 / sqrt(D), as from a head width taken as D / 4 (q doubled:
    exact in bf16)"""
    import synth
    real = o.window_attention

    def doubled(q, k_win, v_win, k_cache, v_cache, cu_rows, prefix_len, suffix=None):
        q2 = synth.f32_to_bf16_bits((o.bf16(q) * 2.0).astype(np.float32))
        return real(q2, k_win, v_win, k_cache, v_cache, cu_rows, prefix_len, suffix)
    monkeypatch.setattr(o, "window_attention", doubled)
    assert _some_pin_fails([ta.test_matches_torch_sdpa])


def test_dropped_prefix_key_is_caught(monkeypatch):
    real = o.window_attention

    def short(q, k_win, v_win, k_cache, v_cache, cu_rows, prefix_len, suffix=None):
        pl = np.maximum(np.asarray(prefix_len) - 1, 0)
        return real(q, k_win, v_win, k_cache, v_cache, cu_rows, pl, suffix)
    monkeypatch.setattr(o, "window_attention", short)
    assert _some_pin_fails([ta.test_matches_torch_sdpa, ta.test_ragged_prefix_and_batch_separation])


def test_round_robin_gqa_is_caught(monkeypatch):
    real = o.window_attention

    def round_robin(q, k_win, v_win, k_cache, v_cache, cu_rows, prefix_len, suffix=None):
        Hq, Hkv = q.shape[1], k_win.shape[1]
        # query head h reads kv head h % Hkv: permute q so that the grouped
        # mapping of the real routine becomes the round-robin one
        perm = np.array([(h % Hkv) * (Hq // Hkv) + h // Hkv for h in range(Hq)])
        out = real(q[:, np.argsort(perm)], k_win, v_win, k_cache, v_cache, cu_rows, prefix_len, suffix)
        return out[:, perm]
    monkeypatch.setattr(o, "window_attention", round_robin)
    assert _some_pin_fails([ta.test_gqa_head_mapping])


def test_maxgap_cut_at_equal_gap_is_caught(monkeypatch):
    real = o.max_gap_filter
    monkeypatch.setattr(o, "max_gap_filter", lambda C, g: real(C, g - 1))
    assert _some_pin_fails([td.test_maxgap_golden, td.test_select_golden])


def test_fallback_of_l_min_rows_is_caught(monkeypatch):
    real = o.select_block

    def fallback_l_min(pos, M, O, argmax, prm):
        return real(pos, M, O, argmax, o.DecisionParams(
            tau=prm.tau, tau_psi=prm.tau_psi, l_min=prm.l_min, l_b=prm.l_min, g_max=prm.g_max,
            eos_id=prm.eos_id, lps_enabled=prm.lps_enabled))
    monkeypatch.setattr(o, "select_block", fallback_l_min)
    assert _some_pin_fails([td.test_select_golden])


def test_strict_kappa_threshold_is_caught(monkeypatch):
    real = o.decide_sequence

    def strict(pos, mask, tokens, in_block, meta, st, w_emb, W, prm, **kw):
        p2 = o.DecisionParams(tau=np.nextafter(prm.tau, np.inf), tau_psi=prm.tau_psi, l_min=prm.l_min,
                              l_b=prm.l_b, g_max=prm.g_max, eos_id=prm.eos_id,
                              lps_enabled=prm.lps_enabled)
        return real(pos, mask, tokens, in_block, meta, st, w_emb, W, p2, **kw)
    monkeypatch.setattr(o, "decide_sequence", strict)
    if not _some_pin_fails([td.test_accept_golden]):
        pytest.fail("no accept pin has kappa exactly at tau")


def _router_pins():
    return [tr.test_lbs_layer_matches_torch_post_norm, tr.test_lps_block_matches_torch_pre_norm,
            tr.test_elementary_layers_match_torch]


def test_router_pins_pass_as_they_stand():
    assert not _some_pin_fails(_router_pins())


def test_tanh_gelu_is_caught(monkeypatch):
    import math

    def tanh_gelu(x):
        return 0.5 * x * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (x + 0.044715 * x ** 3)))
    monkeypatch.setattr(o, "gelu", tanh_gelu)
    assert _some_pin_fails(_router_pins())


def test_layer_norm_eps_is_caught(monkeypatch):
    monkeypatch.setattr(o, "LN_EPS", 1e-6)
    assert _some_pin_fails(_router_pins())


def test_router_attention_scale_is_caught(monkeypatch):
    real = o.softmax_rows
    state = {}

    def wrong_scale(s):  # the scores of a head of width d / heads, rescaled as if by 1/sqrt(d)
        return real(s * state.get("f", 1.0))

    real_attn = o.self_attention

    def attn(x, W, name, n_heads):
        state["f"] = 1.0 / np.sqrt(n_heads)
        try:
            return real_attn(x, W, name, n_heads)
        finally:
            state["f"] = 1.0
    monkeypatch.setattr(o, "softmax_rows", wrong_scale)
    monkeypatch.setattr(o, "self_attention", attn)
    assert _some_pin_fails(_router_pins())


def test_eos_kept_among_candidates_is_caught(monkeypatch):
    real = o.select_block

    def keep_eos(pos, M, O, argmax, prm):
        return real(pos, M, O, argmax, o.DecisionParams(
            tau=prm.tau, tau_psi=prm.tau_psi, l_min=prm.l_min, l_b=prm.l_b, g_max=prm.g_max,
            eos_id=-123456, lps_enabled=prm.lps_enabled))
    monkeypatch.setattr(o, "select_block", keep_eos)
    assert _some_pin_fails([td.test_select_golden])


def test_suffix_one_position_late_is_caught(monkeypatch):
    real = o.window_attention

    def late(q, k_win, v_win, k_cache, v_cache, cu_rows, prefix_len, suffix=None):
        if suffix is not None:
            suffix = np.asarray(suffix).copy()
            suffix[:, 0] += 1
        return real(q, k_win, v_win, k_cache, v_cache, cu_rows, prefix_len, suffix)
    monkeypatch.setattr(o, "window_attention", late)
    assert _some_pin_fails([ta.test_suffix_matches_torch_sdpa, ta.test_suffix_keys_count_once_in_any_order])


def test_append_of_masked_rows_is_caught(monkeypatch):
    real = o.kv_append
    monkeypatch.setattr(o, "kv_append", lambda kc, vc, kw, vw, cu, row_pos, mask:
                        real(kc, vc, kw, vw, cu, row_pos, np.zeros_like(mask)))
    assert _some_pin_fails([ta.test_kv_append_writes_committed_rows_only])


# ---------------------------------------------------------------- router inputs
def _input_pins():
    return [td.test_lps_feature_tuple_golden, tr.test_lps_router_matches_torch_modules,
            tr.test_lbs_router_matches_torch_modules]


def test_input_pins_pass_as_they_stand():
    assert not _some_pin_fails(_input_pins())


@pytest.mark.parametrize("order", [(1, 0, 2, 3, 4), (0, 1, 2, 4, 3), (4, 0, 1, 2, 3)])
def test_lps_features_in_another_order_are_caught(monkeypatch, order):
    real = o.lps_features

    def reordered(pos, mask, in_block, meta, st):
        BM, feats = real(pos, mask, in_block, meta, st)
        return BM, [tuple(f[k] for k in order) for f in feats]
    monkeypatch.setattr(o, "lps_features", reordered)
    assert _some_pin_fails([td.test_lps_feature_tuple_golden])


def test_pos_over_the_masked_count_is_caught(monkeypatch):
    """pos = (i - b) / |B n M| instead of / |B|"""
    real = o.lps_features

    def pos_masked(pos, mask, in_block, meta, st):
        BM, feats = real(pos, mask, in_block, meta, st)
        return BM, [f[:4] + (f[4] * int(meta[1]) / len(BM),) for f in feats]
    monkeypatch.setattr(o, "lps_features", pos_masked)
    assert _some_pin_fails([td.test_lps_feature_tuple_golden])


def test_rho_over_the_window_is_caught(monkeypatch):
    """rho = |M| / window rows (a window-wide mask ratio) instead of |B n M| / |B|"""
    real = o.lps_features

    def rho_window(pos, mask, in_block, meta, st):
        BM, feats = real(pos, mask, in_block, meta, st)
        rho = float(np.count_nonzero(mask)) / len(mask)
        return BM, [f[:3] + (rho, f[4]) for f in feats]
    monkeypatch.setattr(o, "lps_features", rho_window)
    assert _some_pin_fails([td.test_lps_feature_tuple_golden])


def test_gelu_before_layer_norm_in_the_lps_input_is_caught(monkeypatch):
    monkeypatch.setattr(o, "lps_input", lambda x, W: o.layer_norm(
        o.gelu(o.linear(x, W, "lps.in")), W["lps.in_ln.g"], W["lps.in_ln.b"]))
    assert _some_pin_fails(_input_pins())


def _lbs_parts(ent_norm_seq, xhat_seq, w_emb, W, ent_order="lin-gelu-lin-ln"):
    Ht = np.asarray(ent_norm_seq, dtype=np.float64)[:, None]
    if ent_order == "lin-gelu-lin-ln":
        e = o.layer_norm(o.linear(o.gelu(o.linear(Ht, W, "lbs.ent1")), W, "lbs.ent2"),
                         W["lbs.ent_ln.g"], W["lbs.ent_ln.b"])
    else:  # LayerNorm and GELU swapped
        e = o.gelu(o.linear(o.layer_norm(o.linear(Ht, W, "lbs.ent1"), W["lbs.ent_ln.g"],
                                         W["lbs.ent_ln.b"]), W, "lbs.ent2"))
    t = o.linear(o.bf16(w_emb[np.asarray(xhat_seq, dtype=np.int64)]), W, "lbs.tok")
    return e, t


def test_token_branch_first_in_the_fusion_is_caught(monkeypatch):
    """[t ; e] instead of [e ; t] (Eq. lbs_feat)"""
    def swapped(h, x, w_emb, W):
        e, t = _lbs_parts(h, x, w_emb, W)
        return o.linear(np.concatenate([t, e], axis=1), W, "lbs.comb") + W["lbs.pos"][:len(h)]
    monkeypatch.setattr(o, "lbs_input", swapped)
    assert _some_pin_fails(_input_pins())


def test_position_table_before_the_fusion_is_caught(monkeypatch):
    """W_combine([e ; t] + E_pos) instead of W_combine [e ; t] + E_pos"""
    def pos_first(h, x, w_emb, W):
        e, t = _lbs_parts(h, x, w_emb, W)
        return o.linear(np.concatenate([e, t], axis=1) + W["lbs.pos"][:len(h)], W, "lbs.comb")
    monkeypatch.setattr(o, "lbs_input", pos_first)
    assert _some_pin_fails(_input_pins())


def test_layer_norm_and_gelu_swapped_in_the_entropy_branch_are_caught(monkeypatch):
    def swapped(h, x, w_emb, W):
        e, t = _lbs_parts(h, x, w_emb, W, ent_order="lin-ln-lin-gelu")
        return o.linear(np.concatenate([e, t], axis=1), W, "lbs.comb") + W["lbs.pos"][:len(h)]
    monkeypatch.setattr(o, "lbs_input", swapped)
    assert _some_pin_fails(_input_pins())


# ---------------------------------------------------------------- vocabulary ranges
def _range_pins():
    return [lambda: ts.test_range_states_merge_to_the_whole_row(3),
            ts.test_range_state_single_entry_ranges]


def test_range_pins_pass_as_they_stand():
    assert not _some_pin_fails(_range_pins())


def test_merge_without_the_recentring_term_is_caught(monkeypatch):
    """T merged as sum exp(m_g - M) T_g, dropping (m_g - M) S_g"""
    real = o.merge_range_states

    def no_shift(states, V):
        shifted = []
        M = np.stack([s.m for s in states]).max(axis=0)
        for s in states:  # fold the dropped term back out of T so the merge loses it
            shifted.append(o.RangeState(m=s.m, S=s.S, T=s.T - (s.m - M) * s.S, l2=s.l2, idx=s.idx))
        return real(shifted, V)
    monkeypatch.setattr(o, "merge_range_states", no_shift)
    assert _some_pin_fails(_range_pins())


def test_second_logit_from_the_argmax_range_only_is_caught(monkeypatch):
    """l2 taken from the argmax range alone, ignoring the other ranges' maxima"""
    real = o.merge_range_states

    def l2_local(states, V):
        st = real(states, V)
        m = np.stack([s.m for s in states])
        win = np.argmax(m, axis=0)
        l2 = np.array([states[win[r]].l2[r] for r in range(m.shape[1])])
        p2 = np.exp(l2 - m.max(axis=0)) * st.conf
        return o.RowStats(conf=st.conf, entropy=st.entropy, ent_norm=st.ent_norm, gap=st.conf - p2,
                          argmax=st.argmax, logit_gap=st.logit_gap, near_tie=st.near_tie)
    monkeypatch.setattr(o, "merge_range_states", l2_local)
    assert _some_pin_fails(_range_pins())
