"""ebd_lm_stats_noalloc (allocation-free LM-head statistics, scratch in a
static device array) against the handle path ebd_lm_stats: two calls in a
row on the same scratch, different inputs and row counts, bit-identical
statistics.  Also checks the statistics against the oracle on a few rows and
the size limit.  Runs alone or after the other GPU tests."""
import numpy as np
import pytest

import synth
from oracle import ebd_oracle as o
from tests import parity

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

# 32000 / 64 = 500 vocabulary units: more than the SMs, so every CTA of the
# persistent LM head leaves a partial of every row in the scratch
SHAPE = synth.tiny.with_(name="noalloc", d_model=1024, vocab=32000, n_heads_q=8, n_heads_kv=8,
                         head_dim=128, prefix=16, windows=(64,), seed=11)
KEYS = ("conf", "entropy", "ent_norm", "gap", "argmax")


def _outputs(rows):
    f32 = dict(dtype=torch.float32, device="cuda")
    out = {k: torch.full((rows,), float("nan"), **f32) for k in KEYS[:4]}
    out["argmax"] = torch.full((rows,), -7, dtype=torch.int32, device="cuda")
    return out


def _noalloc(E, hidden, w, rows, status):
    out = _outputs(rows)
    s = E.ebd_lm_stats_noalloc(hidden.data_ptr(), w.w_lm.data_ptr(), w.layout, rows,
                               SHAPE.d_model, SHAPE.vocab, out["conf"].data_ptr(),
                               out["entropy"].data_ptr(), out["ent_norm"].data_ptr(),
                               out["gap"].data_ptr(), out["argmax"].data_ptr(),
                               status.data_ptr(), torch.cuda.current_stream().cuda_stream)
    assert s == E.EBD_OK
    return out


def _handle_path(E, rt, h, hidden, w, rows):
    out = _outputs(rows)
    a = E.ebd_step_args()
    a.batch, a.rows = 1, rows
    a.hidden = hidden.data_ptr()
    a.w_lm = w.w_lm.data_ptr()
    a.w_lm_layout = w.layout
    for k in KEYS:
        setattr(a, k, out[k].data_ptr())
    E.check(E.ebd_lm_stats(h.h, a, rt.stream_handle(None)), h.h)
    assert h.sync_status() == 0
    return out


@pytest.mark.parametrize("layout", ["rowmajor", "packed"])
def test_noalloc_matches_handle_path_twice_in_a_row(layout):
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    inp = synth.make_step_inputs(SHAPE)
    w = rt.upload_weights(inp)
    h = rt.Handle(rt.config_for(SHAPE))
    if layout == "packed":
        w = rt.pack_weights(h, w)
    hid_all = synth.bf16_to_f32(inp.hidden).reshape(inp.rows, -1)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    try:
        # call 1: all 64 rows (the maximum); call 2: 17 rows of other hidden
        # states, so a partial left over from call 1 would show
        cases = [(64, hid_all), (17, hid_all[::-1][:17] * 0.75)]
        for rows, hid in cases:
            hidden = rt._dev(synth.f32_to_bf16_bits(np.ascontiguousarray(hid)), "cuda")
            got = _noalloc(E, hidden, w, rows, status)
            torch.cuda.synchronize()
            assert int(status.item()) == 0
            ref = _handle_path(E, rt, h, hidden, w, rows)
            for k in KEYS:
                np.testing.assert_array_equal(got[k].cpu().numpy(), ref[k].cpu().numpy(), err_msg=k)
            # and the statistics themselves, on a few rows, against the oracle
            # (lm_logits takes bf16 bit patterns)
            bits = synth.f32_to_bf16_bits(np.ascontiguousarray(hid))
            sample = [0, rows // 2, rows - 1]
            st = o.softmax_stats(o.lm_logits(bits[sample],
                                             inp.w_lm.reshape(SHAPE.vocab, SHAPE.d_model)))
            parity.compare_stats(st, {k: got[k].cpu().numpy()[sample] for k in KEYS})
    finally:
        h.close()


def test_noalloc_rejects_sizes_beyond_the_maximum():
    from paper_2609_16450_gb300 import _ebd as E
    big = E.EBD_NOALLOC_MAX_ROWS + 1
    buf = torch.zeros(big * SHAPE.d_model, dtype=torch.int16, device="cuda")
    w = torch.zeros(SHAPE.vocab * SHAPE.d_model, dtype=torch.int16, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    s = E.ebd_lm_stats_noalloc(buf.data_ptr(), w.data_ptr(), 0, big, SHAPE.d_model, SHAPE.vocab,
                               0, 0, 0, 0, 0, status.data_ptr(), 0)
    assert s == E.EBD_ERR_UNSUPPORTED
    s = E.ebd_lm_stats_noalloc(buf.data_ptr(), w.data_ptr(), 0, 4, SHAPE.d_model, SHAPE.vocab,
                               0, 0, 0, 0, 0, 0, 0)
    assert s == E.EBD_ERR_INVALID_ARG  # no status word
    assert E.ebd_lm_stats_noalloc(buf.data_ptr(), w.data_ptr(), 0, 0, SHAPE.d_model, SHAPE.vocab,
                                  0, 0, 0, 0, 0, status.data_ptr(), 0) == E.EBD_OK
