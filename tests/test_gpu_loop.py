"""The generation loop (App. E algorithm, block-forward windows of Sec. 6.4)
on the GPU through the C ABI, against the oracle's loop.

At the tiny loop shape the oracle runs the whole loop: windows, accepted
sets, committed tokens and attention outputs must match step by step up to
the first step the oracle flags for a near-tie (after which the two runs may
legitimately part).  At the LLaDA-8B loop shape the GPU loop runs to the end
and every step's decision is checked against the oracle's decision on the
GPU's statistics, the statistics themselves on sampled rows, and the loop
invariants throughout."""
import numpy as np
import pytest

import synth
from oracle import ebd_oracle as o
from tests import parity

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


def _prm(sh):
    return o.DecisionParams(tau=sh.tau, tau_psi=sh.tau_psi, l_min=sh.l_min, l_b=sh.l_b,
                            g_max=sh.g_max, eos_id=sh.eos_id, lps_enabled=bool(sh.lps_enabled))


def _gpu_loop(sh, inp, attention=True, packed=False):
    from paper_2609_16450_gb300 import loop as lp
    from paper_2609_16450_gb300 import runtime as rt
    w = rt.upload_weights(inp)
    h = rt.Handle(lp.config_for_loop(sh), w.w_emb)
    if packed:
        w = rt.pack_weights(h, w)
    try:
        return lp.run_loop(h, sh, w, lambda s, p: synth.loop_window_inputs(sh, s, p),
                           lambda p: synth.loop_kv(sh, p), attention=attention)
    finally:
        h.close()


def _check_invariants(sh, res):
    L = sh.gen_len
    assert res.steps <= L
    assert all(c >= 1 for c in res.commits), "a step committed nothing"
    assert sum(res.commits) == L
    assert np.all(res.tokens >= 0) and np.all(res.tokens < sh.vocab)
    for r in res.records:
        lo, hi = r.window
        acc = r.accepted.astype(bool)
        assert np.all(r.before["mask"][acc] == 1), "commit of an unmasked row"
        assert np.all(r.after["tokens"][acc] == r.argmax[acc]), "commit value != x_hat"
        assert np.all(r.after["mask"][acc] == 0)
        assert np.array_equal(r.after["mask"][~acc], r.before["mask"][~acc])


def test_loop_tiny_matches_oracle():
    sh = synth.loop_tiny
    inp = synth.make_step_inputs(sh)
    res = _gpu_loop(sh, inp)
    _check_invariants(sh, res)
    W = o.weights_f64(synth.router_weights(sh.seed, sh.d_base, sh.gen_len))
    toks, steps, commits, recs = o.generation_loop(
        sh, W, _prm(sh), lambda s, p: synth.loop_window_inputs(sh, s, p),
        lambda p: synth.loop_kv(sh, p), inp.w_lm, inp.w_emb, attention=True)
    compared = 0
    prm = _prm(sh)
    for g in res.records:  # every GPU step is the rules' decision on its own features
        lo, hi = g.window
        b = g.before
        out = {"conf": g.conf, "argmax": g.argmax, "lbs_logit": g.lbs_logit,
               "lps_prob": g.lps_prob, "accepted": g.accepted, "tokens": g.after["tokens"],
               "mask": g.after["mask"], "in_block": g.after["in_block"]}
        parity.check_decision_valid(sh.prefix + np.arange(lo, hi), b["mask"], b["tokens"],
                                    b["in_block"], b["meta"], out, g.after["meta"], prm)
    first_flag = None
    for g, r in zip(res.records, recs):
        assert g.window == r["window"], (g.step, g.window, r["window"])
        parity._close(f"attn step {g.step}", g.attn_out, r["attn"])
        st = r["stats"]
        for k in ("conf", "entropy", "gap"):
            parity._close(f"{k} step {g.step}", getattr(g, k), getattr(st, k))
        nt = st.near_tie
        assert np.array_equal(g.argmax[~nt], st.argmax[~nt]), g.step
        if r["flag"] or r["flag_lbs"]:
            first_flag = g.step
            break  # a near-tie decision: the runs may part from here
        assert np.array_equal(g.accepted, r["accepted"]), (g.step, g.accepted, r["accepted"])
        compared += 1
    else:
        assert res.steps == steps
        ties = np.zeros(sh.gen_len, bool)
        for g, r in zip(res.records, recs):
            lo, hi = g.window
            ties[lo:hi] |= r["stats"].near_tie & r["accepted"].astype(bool)
        assert np.array_equal(res.tokens[~ties], toks[~ties])
    print("steps", res.steps, "oracle", steps, "compared", compared, "first flagged", first_flag)
    # every step up to the first flagged one (or all of them) was compared
    assert compared == (res.steps if first_flag is None else first_flag)
    assert compared >= min(10, res.steps)


def test_loop_llada_full_size():
    sh = synth.loop_shape
    inp = synth.make_step_inputs(sh)
    res = _gpu_loop(sh, inp, packed=True)
    _check_invariants(sh, res)
    W = o.weights_f64(synth.router_weights(sh.seed, sh.d_base, sh.gen_len))
    prm = _prm(sh)
    flagged = 0
    for g in res.records:
        lo, hi = g.window
        R = hi - lo
        st = o.RowStats(conf=g.conf.astype(np.float64), entropy=g.entropy.astype(np.float64),
                        ent_norm=g.ent_norm.astype(np.float64), gap=g.gap.astype(np.float64),
                        argmax=g.argmax.astype(np.int64), logit_gap=np.full(R, np.inf),
                        near_tie=np.zeros(R, bool))
        b = g.before
        t, m, ib, meta = b["tokens"].copy(), b["mask"].copy(), b["in_block"].copy(), b["meta"].copy()
        d = o.decide_sequence(sh.prefix + np.arange(lo, hi), m, t, ib, meta, st, inp.w_emb, W, prm)
        if d.flag_accept or d.flag_lbs:
            flagged += 1
            out = {"conf": g.conf, "argmax": g.argmax, "lbs_logit": g.lbs_logit,
                   "lps_prob": g.lps_prob, "accepted": g.accepted, "tokens": g.after["tokens"],
                   "mask": g.after["mask"], "in_block": g.after["in_block"]}
            parity.check_decision_valid(sh.prefix + np.arange(lo, hi), b["mask"], b["tokens"],
                                        b["in_block"], b["meta"], out, g.after["meta"], prm)
            continue
        a = g.after
        assert np.array_equal(g.accepted, d.accepted), g.step
        assert np.array_equal(a["mask"], m) and np.array_equal(a["tokens"], t), g.step
        assert np.array_equal(a["in_block"], ib) and np.array_equal(a["meta"], meta), g.step
    # the statistics of two rows at the first, middle and last step
    for g in (res.records[0], res.records[len(res.records) // 2], res.records[-1]):
        lo, hi = g.window
        pos = sh.prefix + np.arange(lo, hi, dtype=np.int32)
        hid = synth.loop_window_inputs(sh, g.step, pos)[0]
        rows = np.array(sorted({0, hi - lo - 1}))
        st = o.softmax_stats(o.lm_logits(hid[rows], inp.w_lm))
        parity.compare_stats(st, {"conf": g.conf[rows], "entropy": g.entropy[rows],
                                  "ent_norm": g.ent_norm[rows], "gap": g.gap[rows],
                                  "argmax": g.argmax[rows]})
    print("steps", res.steps, "flagged", flagged, "device us", round(res.device_us, 1))
    assert flagged <= res.steps // 4
