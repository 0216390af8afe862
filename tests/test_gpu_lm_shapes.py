"""The LM head's launch shapes at their boundaries, every row against the
oracle, through ebd_lm_stats: one CTA per SM below 65 rows, CTA pairs
(cta_group::2) from 65 rows, two row groups above 432 rows, two N sub-tiles
between 257 and 432 rows; a vocabulary that ends in a partial 64-row unit
(4000 entries); both W layouts; and vocabulary shards so small that the odd
CTA of a pair has no W rows in some chunks (ebd_lm_shard_state)."""
import numpy as np
import pytest

import synth
from oracle import ebd_oracle as o
from tests import parity

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

KEYS = ("conf", "entropy", "ent_norm", "gap", "argmax")


def _shape(rows, vocab):
    return synth.tiny.with_(name=f"lm_{rows}_{vocab}", vocab=vocab, windows=(rows,),
                            gen_len=max(512, rows), prefix=0)


def _run(sh, layout, shards=1):
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    from paper_2609_16450_gb300 import vocab_parallel as vp
    inp = synth.make_step_inputs(sh)
    R = inp.rows
    w = rt.upload_weights(inp)
    h = rt.Handle(rt.config_for(sh, max_window=R, max_rows=R))
    try:
        if layout == "packed":
            w = rt.pack_weights(h, w)
        hidden = rt._dev(inp.hidden, "cuda")
        out = {k: torch.empty(R, dtype=torch.int32 if k == "argmax" else torch.float32,
                              device="cuda") for k in KEYS}
        a = E.ebd_step_args()
        a.batch, a.rows = 1, R
        a.hidden, a.w_lm, a.w_lm_layout = hidden.data_ptr(), w.w_lm.data_ptr(), w.layout
        for k in KEYS:
            setattr(a, k, out[k].data_ptr())
        if shards == 1:
            E.check(E.ebd_lm_stats(h.h, a, rt.stream_handle(None)), h.h)
        else:
            states = torch.empty((shards, R, vp.STATE_WORDS), dtype=torch.float32, device="cuda")
            for g in range(shards):
                v0, v1 = vp.shard_range(sh.vocab, shards, g)
                s = E.ebd_step_args()
                s.batch, s.rows, s.hidden, s.w_lm_layout = 1, R, hidden.data_ptr(), w.layout
                s.w_lm = vp.shard_weights(w.w_lm, sh.vocab, sh.d_model, v0, v1, w.layout).data_ptr()
                E.check(E.ebd_lm_shard_state(h.h, s, v0, v1 - v0, states[g].data_ptr(),
                                             rt.stream_handle(None)), h.h)
            E.check(E.ebd_merge_shard_states(h.h, states.data_ptr(), shards, a,
                                             rt.stream_handle(None)), h.h)
        assert h.sync_status() == 0, E.ebd_last_error(h.h)
        torch.cuda.synchronize()
        got = {k: v.cpu().numpy() for k, v in out.items()}
    finally:
        h.close()
    st = o.softmax_stats(o.lm_logits(inp.hidden.reshape(R, -1), inp.w_lm.reshape(sh.vocab, -1)))
    return parity.compare_stats(st, got)


@pytest.mark.parametrize("rows", [64, 65, 100, 256, 257, 300, 432, 433, 512])
@pytest.mark.parametrize("vocab", [4096, 4000])
def test_lm_head_launch_shapes(rows, vocab):
    rep = _run(_shape(rows, vocab), "packed" if rows % 2 else "rowmajor")
    assert rep["conf"] <= 2e-3


@pytest.mark.parametrize("rows,shards", [(100, 16), (100, 32), (512, 32), (32, 7)])
def test_small_vocabulary_shards(rows, shards):
    """4096 / shards vocabulary rows per shard: 4 or 2 units, i.e. one chunk
    per pair, whose odd CTA holds no W rows at 2 units; and 7 uneven shards
    of the one-CTA-per-SM launch."""
    _run(_shape(rows, 4096), "packed", shards=shards)
    _run(_shape(rows, 4096), "rowmajor", shards=shards)
