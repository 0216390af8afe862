"""Guard words around every buffer a step writes (outputs, decode state,
K/V cache with the append), checked after steps of the tiny, LLaDA-8B and
Dream-7B shapes, with and without an active block, on the cluster and the
grid-wide decision paths and, forced with EBD_DECIDE_KERNEL, on the one-CTA
decision kernel."""
import contextlib
import os

import numpy as np
import pytest

import synth
from tests import guards

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

# (shape, state, window attention, cache append, decision kernel forced or "")
CASES = [("tiny", "select", True, False, ""), ("tiny", "inblock", True, True, ""),
         ("llada8b", "select", True, False, ""), ("dream7b", "select", True, True, ""),
         ("tiny_full", "select", False, False, ""), ("tiny_full", "inblock", False, False, ""),
         ("tiny", "select", True, False, "cta"), ("tiny", "inblock", True, True, "cta"),
         ("llada8b", "select", True, False, "cta")]


@contextlib.contextmanager
def decide_kernel(kernel):
    """EBD_DECIDE_KERNEL set to `kernel` (unset for "") inside the block."""
    old = os.environ.pop("EBD_DECIDE_KERNEL", None)
    if kernel:
        os.environ["EBD_DECIDE_KERNEL"] = kernel
    try:
        yield
    finally:
        os.environ.pop("EBD_DECIDE_KERNEL", None)
        if old is not None:
            os.environ["EBD_DECIDE_KERNEL"] = old


@pytest.mark.parametrize("name,state,attention,append,kernel", CASES)
def test_step_writes_stay_inside_its_buffers(name, state, attention, append, kernel):
    with decide_kernel(kernel):
        _guarded(name, state, attention, append)


def _guarded(name, state, attention, append):
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    sh = synth.SHAPES[name]
    inp = synth.make_step_inputs(sh)
    if state == "inblock":
        synth.preset_in_block(inp, 20)
    w = rt.upload_weights(inp)
    h = rt.Handle(rt.config_for(sh), w.w_emb)
    try:
        if name != "tiny":
            w = rt.pack_weights(h, w)
        status, out, g = guards.guarded_step(E, rt, h, inp, w, attention=attention, append=append)
        assert status == 0, E.ebd_last_error(h.h)
        broken = [k for k, v in g.items() if not v.intact()]
        assert not broken, f"guard words overwritten around {broken}"
        assert np.isfinite(out["conf"]).all() and (out["argmax"] >= 0).all()
        assert out["accepted"].sum() >= 1
    finally:
        h.close()
