"""The GPU parity checker itself, on the CPU: the oracle's own decisions,
presented as if they came from the GPU, pass tests/parity.py's checks
(including the validity re-derivation that flagged sequences rely on), and
planted faults in them (an extra commit, a changed uncommitted token, a
wrong block state, a dropped commit) are caught."""
import numpy as np
import pytest

import synth
from oracle import ebd_oracle as o
from tests import parity


def _prm(sh):
    return o.DecisionParams(tau=sh.tau, tau_psi=sh.tau_psi, l_min=sh.l_min, l_b=sh.l_b,
                            g_max=sh.g_max, eos_id=sh.eos_id, lps_enabled=bool(sh.lps_enabled))


def _as_gpu(res):
    return dict(conf=res.stats.conf.astype(np.float32), argmax=res.stats.argmax.astype(np.int32),
                lbs_logit=res.lbs_logit.astype(np.float32), lps_prob=res.lps_prob.astype(np.float32),
                accepted=res.accepted.copy(), tokens=res.tokens.copy(), mask=res.mask.copy(),
                in_block=res.in_block.copy(), blk_meta=res.blk_meta.copy())


_cases = {}


def _case(name, state):
    key = (name, state)
    if key not in _cases:
        sh = synth.SHAPES[name]
        inp = synth.make_step_inputs(sh)
        if state == "inblock":
            synth.preset_in_block(inp, 20)
        W = o.weights_f64(synth.router_weights(sh.seed, sh.d_base, sh.gen_len))
        _cases[key] = (sh, inp, o.step(inp, W, _prm(sh), attention=False))
    return _cases[key]


@pytest.mark.parametrize("name", ["tiny", "tiny_full"])
@pytest.mark.parametrize("state", ["select", "inblock"])
def test_oracle_decisions_pass_the_checker(name, state):
    sh, inp, res = _case(name, state)
    rep = parity.compare_decision(res, _as_gpu(res), inp, _prm(sh))
    assert rep["sequences"] == sh.batch


def _fails(sh, inp, res, gpu):
    try:
        parity.compare_decision(res, gpu, inp, _prm(sh))
    except AssertionError:
        return True
    return False


@pytest.mark.parametrize("state", ["select", "inblock"])
def test_planted_faults_are_caught(state):
    sh, inp, res = _case("tiny_full", state)
    # flag every sequence, so only the validity re-derivation can catch them
    res_f = o.StepResult(**{**res.__dict__, "flag_accept": np.ones_like(res.flag_accept)})
    base = _as_gpu(res)
    assert not _fails(sh, inp, res_f, base)
    acc = np.flatnonzero(base["accepted"])
    masked_not_acc = np.flatnonzero((inp.mask == 1) & (base["accepted"] == 0))
    assert acc.size and masked_not_acc.size
    g = {k: v.copy() for k, v in base.items()}           # an extra commit
    r = masked_not_acc[0]
    g["accepted"][r] = 1; g["mask"][r] = 0; g["tokens"][r] = g["argmax"][r]
    assert _fails(sh, inp, res_f, g)
    g = {k: v.copy() for k, v in base.items()}           # a dropped commit
    r = acc[0]
    g["accepted"][r] = 0; g["mask"][r] = 1; g["tokens"][r] = inp.tokens[r]
    assert _fails(sh, inp, res_f, g)
    g = {k: v.copy() for k, v in base.items()}           # an uncommitted token changed
    r = np.flatnonzero(base["accepted"] == 0)[0]
    g["tokens"][r] = (g["tokens"][r] + 1) % sh.vocab
    assert _fails(sh, inp, res_f, g)
    g = {k: v.copy() for k, v in base.items()}           # a wrong block state
    b = int(np.flatnonzero(base["blk_meta"][:, 1] > 0)[0])
    g["blk_meta"][b, 1] += 1
    assert _fails(sh, inp, res_f, g)
