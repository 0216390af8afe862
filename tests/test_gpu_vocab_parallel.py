"""GPU parity of the vocabulary-parallel LM head, called through the C ABI
(ebd_lm_shard_state, ebd_merge_shard_states).  The G ranks are emulated on
one GPU as G independent shard launches (none waits on another); their
states are stacked as the all-gather would stack them and merged.  Checked:
the merged statistics against the single launch over the whole vocabulary
(ebd_lm_stats: argmax identical, the floating-point statistics within 1e-5,
the two differing only in the association order of the merge) and against
the oracle; and the decision taken on the merged statistics against the one
taken on the single launch's."""
import numpy as np
import pytest

import synth
from oracle import ebd_oracle as o
from tests import parity

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

KEYS = ("conf", "entropy", "ent_norm", "gap", "argmax")


def _outs(rows):
    f32 = dict(dtype=torch.float32, device="cuda")
    d = {k: torch.empty(max(rows, 1), **f32) for k in KEYS[:-1]}
    d["argmax"] = torch.empty(max(rows, 1), dtype=torch.int32, device="cuda")
    return d


def _args(E, ds, out):
    a = ds.args()
    for k in KEYS:
        setattr(a, k, out[k].data_ptr())
    return a


def _fetch(out, rows):
    torch.cuda.synchronize()
    return {k: v[:rows].cpu().numpy() for k, v in out.items()}


@pytest.mark.parametrize("shape,world,layout", [("tiny", 3, "rowmajor"), ("tiny", 2, "packed"),
                                                ("llada8b", 2, "packed"), ("llada8b", 3, "rowmajor"),
                                                ("dream7b", 4, "packed")])
def test_sharded_statistics_match_the_whole_vocabulary(shape, world, layout):
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    from paper_2609_16450_gb300 import vocab_parallel as vp
    sh = synth.SHAPES[shape]
    inp = synth.make_step_inputs(sh)
    w = rt.upload_weights(inp)
    h = rt.Handle(rt.config_for(sh), w.w_emb)
    try:
        if layout == "packed":
            w = rt.pack_weights(h, w)
        ds = rt.DeviceStep(inp, w, attention=False)
        R = inp.rows
        full = _outs(R)
        E.check(E.ebd_lm_stats(h.h, _args(E, ds, full), rt.stream_handle(None)), h.h)
        ref = _fetch(full, R)
        states = torch.empty((world, R, vp.STATE_WORDS), dtype=torch.float32, device="cuda")
        for g in range(world):  # one launch per emulated rank
            v0, v1 = vp.shard_range(sh.vocab, world, g)
            shard = vp.shard_weights(w.w_lm, sh.vocab, sh.d_model, v0, v1, w.layout)
            a = _args(E, ds, _outs(R))
            a.w_lm = shard.data_ptr()
            E.check(E.ebd_lm_shard_state(h.h, a, v0, v1 - v0, states[g].data_ptr(),
                                         rt.stream_handle(None)), h.h)
        merged = _outs(R)
        a = _args(E, ds, merged)
        E.check(E.ebd_merge_shard_states(h.h, states.data_ptr(), world, a, rt.stream_handle(None)),
                h.h)
        got = _fetch(merged, R)
        assert h.sync_status() == 0
        np.testing.assert_array_equal(got["argmax"], ref["argmax"])
        for k in KEYS[:-1]:
            np.testing.assert_allclose(got[k], ref[k], rtol=0, atol=1e-5, err_msg=k)
        # each shard's argmax lies in its own range
        st = states.cpu().numpy()
        for g in range(world):
            v0, v1 = vp.shard_range(sh.vocab, world, g)
            idx = st[g, :, 4].copy().view(np.int32)
            assert ((idx >= v0) & (idx < v1)).all()
        # against the oracle: every row at the tiny shape, sampled rows otherwise
        rows = np.arange(R) if sh.vocab <= 4096 else np.unique(np.linspace(0, R - 1, 6).astype(int))
        W = inp.w_lm.reshape(sh.vocab, sh.d_model)
        ost = o.softmax_stats(o.lm_logits(inp.hidden.reshape(R, sh.d_model)[rows], W))
        parity.compare_stats(ost, {k: got[k][rows] for k in KEYS})
    finally:
        h.close()


@pytest.mark.parametrize("shape", ["tiny", "llada8b"])
def test_decision_on_merged_statistics(shape):
    """The decision each rank takes on the merged statistics (ebd_decide) is
    the decision on the single launch's statistics."""
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    from paper_2609_16450_gb300 import vocab_parallel as vp
    sh = synth.SHAPES[shape]
    inp = synth.make_step_inputs(sh)
    w = rt.upload_weights(inp)
    h = rt.Handle(rt.config_for(sh), w.w_emb)
    try:
        results = []
        for world in (1, 2):
            ds = rt.DeviceStep(inp, w, attention=False)
            R = inp.rows
            states = torch.empty((world, R, vp.STATE_WORDS), dtype=torch.float32, device="cuda")
            for g in range(world):
                v0, v1 = vp.shard_range(sh.vocab, world, g)
                a = ds.args()
                a.w_lm = vp.shard_weights(w.w_lm, sh.vocab, sh.d_model, v0, v1, w.layout).data_ptr()
                E.check(E.ebd_lm_shard_state(h.h, a, v0, v1 - v0, states[g].data_ptr(),
                                             rt.stream_handle(None)), h.h)
            a = ds.args()
            E.check(E.ebd_merge_shard_states(h.h, states.data_ptr(), world, a,
                                             rt.stream_handle(None)), h.h)
            E.check(E.ebd_decide(h.h, a, rt.stream_handle(None)), h.h)
            assert h.sync_status() == 0
            results.append(ds.fetch())
        one, two = results
        for k in ("tokens", "mask", "in_block", "blk_meta", "accepted", "argmax"):
            np.testing.assert_array_equal(one[k], two[k], err_msg=k)
    finally:
        h.close()


def test_shard_arguments_are_checked():
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    sh = synth.tiny
    inp = synth.make_step_inputs(sh)
    w = rt.upload_weights(inp)
    h = rt.Handle(rt.config_for(sh), w.w_emb)
    try:
        ds = rt.DeviceStep(inp, w, attention=False)
        st = torch.empty((inp.rows, 8), dtype=torch.float32, device="cuda")
        a = ds.args()
        for v0, n in ((32, 64), (0, sh.vocab + 64), (-64, 64), (0, 0)):
            assert E.ebd_lm_shard_state(h.h, a, v0, n, st.data_ptr(), 0) == E.EBD_ERR_INVALID_ARG
        assert E.ebd_merge_shard_states(h.h, st.data_ptr(), 0, a, 0) == E.EBD_ERR_INVALID_ARG
    finally:
        h.close()
