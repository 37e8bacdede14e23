"""The kernels' bounded waits: a wait that runs out ends the launch with a status, not a hang.

kvx_debug_stall_next_translate makes the identity kernel's first CTA stop issuing its source
copies at a chosen work unit, with every on-chip wait bounded at 2 ms.  The launch must come
back (well within a second), record KVX_DEV_WAIT_TIMEOUT, and leave the context usable: the
next call, with the normal bounds, equals the oracle.
"""
import dataclasses
import time

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2608_30963_gb300 as kvx
from paper_2608_30963_gb300 import synth

from harness import compare, make_case, oracle_problem

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("unit", [0, 1])
def test_wait_that_runs_out_returns_a_status_and_the_next_call_is_correct(unit):
    from gpu_harness import DeviceCase
    kvx.build()
    spec = synth.config_specs()["qwen7b_to_qwen1p5b_4k"]
    spec = dataclasses.replace(spec, src=dataclasses.replace(spec.src, num_layers=4),
                               dst=dataclasses.replace(spec.dst, num_layers=4))
    c = make_case(spec, [4096])   # 256 K and 256 V units over the SMs: CTA 0 walks at least two
    g = DeviceCase(c, path=kvx.KVX_PATH_AUTO)
    assert g.tr.device_status() == 0
    g.tr.debug_stall_next_translate(unit, 2000)
    t0 = time.perf_counter()
    g.run()
    torch.cuda.synchronize()
    took = time.perf_counter() - t0
    bits = g.tr.device_status()
    assert bits & kvx.KVX_DEV_WAIT_TIMEOUT, f"status 0x{bits:x}"
    assert took < 1.0, took
    # the context is usable and the next call (normal bounds) is complete and correct
    for t in g.dst_k + g.dst_v:
        t.fill_(float("nan"))
    g.run()
    torch.cuda.synchronize()
    assert g.tr.device_status() == 0
    ok, ov = oracle_problem(c).translate()
    gk, gv = g.gather()
    compare(gk, ok, "bf16", "after a timed-out call K")
    compare(gv, ov, "bf16", "after a timed-out call V")
