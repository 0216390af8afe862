"""Run by tests/test_gpu_checked_build.py in a fresh process whose
EBD_LIBRARY names the checked build (libebd_checked.so, compiled with
-DEBD_CHECKS): the guarded steps of tests/test_gpu_guards.py, whose outputs
are saved for comparison with the normal build, and one window-attention call
whose row offsets overrun the step's rows, which the checked build must
report as EBD_ERR_BOUNDS without writing outside any buffer."""
import sys

import numpy as np


def run_cases():
    import synth
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    from tests import guards
    from tests.test_gpu_guards import CASES, decide_kernel
    res = {}
    for name, state, attention, append, kernel in CASES:
        sh = synth.SHAPES[name]
        inp = synth.make_step_inputs(sh)
        if state == "inblock":
            synth.preset_in_block(inp, 20)
        w = rt.upload_weights(inp)
        h = rt.Handle(rt.config_for(sh), w.w_emb)
        try:
            if name != "tiny":
                w = rt.pack_weights(h, w)
            with decide_kernel(kernel):
                status, out, g = guards.guarded_step(E, rt, h, inp, w, attention=attention,
                                                     append=append)
            key = f"{name}_{state}" + (f"_{kernel}" if kernel else "")
            res[key + "/status"] = np.array(status)
            res[key + "/guards"] = np.array(all(v.intact() for v in g.values()))
            for k, v in out.items():
                res[f"{key}/{k}"] = v
        finally:
            h.close()
    return res


def bounds_case():
    import synth
    from paper_2609_16450_gb300 import _ebd as E
    from paper_2609_16450_gb300 import runtime as rt
    from tests import guards
    sh = synth.tiny
    inp = synth.make_step_inputs(sh)   # cu_rows = [0, 32]
    w = rt.upload_weights(inp)
    h = rt.Handle(rt.config_for(sh), w.w_emb)
    try:
        status, out, g = guards.guarded_step(E, rt, h, inp, w, call="attention", rows=24)
        return {"bounds/status": np.array(status),
                "bounds/guards": np.array(all(v.intact() for v in g.values()))}
    finally:
        h.close()


if __name__ == "__main__":
    from paper_2609_16450_gb300 import _ebd as E
    assert E.load()._name.endswith("libebd_checked.so"), E.load()._name
    res = run_cases()
    res.update(bounds_case())
    np.savez(sys.argv[1], **res)
    print("checked run ok")
