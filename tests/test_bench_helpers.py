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


def test_partials_per_row_rule():
    """The partial states per row a handle keeps: the unpaired grid, or the
    paired one (one pair per two SMs) when a step may take it."""
    b = _bench()
    assert b.lm_pair_grid(152, 1976) == 152 and b.lm_pair_grid(152, 64) == 32
    assert b.partials_per_row(152, 1976, 32) == 142       # LLaDA-8B step: unpaired
    assert b.partials_per_row(152, 2376, 512) == 152      # Dream-7B: pairs possible
    assert b.partials_per_row(152, 64, 512) == 64         # tiny vocabulary


def test_parity_summary_of_the_oracle_itself():
    """bench.py's parity block, given the oracle's own outputs as the GPU's,
    reports no mismatch; a changed argmax and a changed commit are counted."""
    from oracle import ebd_oracle as o
    b = _bench()
    sh = synth.tiny
    inp = synth.make_step_inputs(sh)
    W = o.weights_f64(synth.router_weights(sh.seed, sh.d_base, sh.gen_len))
    prm = o.DecisionParams(tau=sh.tau, tau_psi=sh.tau_psi, l_min=sh.l_min, l_b=sh.l_b,
                           g_max=sh.g_max, eos_id=sh.eos_id, lps_enabled=bool(sh.lps_enabled))
    res = o.step(inp, W, prm)
    gpu = dict(conf=res.stats.conf.astype(np.float32), entropy=res.stats.entropy.astype(np.float32),
               ent_norm=res.stats.ent_norm.astype(np.float32), gap=res.stats.gap.astype(np.float32),
               argmax=res.stats.argmax.astype(np.int32), accepted=res.accepted.copy(),
               tokens=res.tokens.copy(), mask=res.mask.copy(), in_block=res.in_block.copy(),
               blk_meta=res.blk_meta.copy(), attn_out=res.attn_out.astype(np.float32))
    rep = b.parity_summary(sh, inp, res, gpu)
    assert rep["argmax_mismatch"] == 0 and not any(rep["decision_mismatch"].values())
    assert rep["within_tolerance"] and rep["max_abs_diff"]["conf"] < 1e-6
    assert set(rep["near_ties"]) == {"top2_logit_gap", "kappa_vs_tau", "p_psi_vs_tau_psi",
                                     "lbs_logit_vs_0"}
    r = int(np.flatnonzero(~res.stats.near_tie)[0])
    gpu["argmax"][r] += 1
    acc = int(np.flatnonzero(res.accepted)[0])
    gpu["accepted"][acc] = 0
    rep = b.parity_summary(sh, inp, res, gpu)
    assert rep["argmax_mismatch"] == 1
    if rep["flagged_sequences"] == 0:
        assert rep["decision_mismatch"]["accepted"] == 1 and not rep["within_tolerance"]


def test_kernel_hash_ignores_comments_only():
    """The profiled-traffic hash follows the LM head's code, not its
    comments: a comment-only change keeps it, a code change does not."""
    b = _bench()
    import os as _os
    base = lambda f: open(_os.path.join(ROOT, "paper_2609_16450_gb300", "csrc", f)).read()
    h0 = b.lm_kernel_hash(base)
    assert b.lm_kernel_hash(lambda f: "// a note\n/* and\n another */\n" + base(f) + "\n// end\n") == h0
    assert b.lm_kernel_hash(lambda f: base(f).replace("kUnit", "kUnit ", 1) + "\nint x;\n") != h0


def test_headline_profile_matches_the_lm_head_sources():
    """The committed ncu capture of the headline LM head was taken on the
    current LM-head sources (else bench.py reports no traffic): a code change
    to k_lmhead.cu, ptx.cuh or lm_params.h needs a new capture."""
    b = _bench()
    t = b.profiled_traffic("llada8b")
    assert t is not None and t > 1.0e9
