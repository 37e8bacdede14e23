"""Writes oracle_regression.json: sampled outputs of the oracle (`oracle/`) on small seeded
cases, so that any later change to the oracle's arithmetic shows up as a test failure and has
to be justified.  It calls only the oracle, through the test harness, on inputs from the
seeded generator.

    python tests/golden/make_oracle_golden.py
"""
import dataclasses
import json
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(HERE))                     # tests/ (harness)
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))    # repository root

from harness import make_case, oracle_problem  # noqa: E402
from paper_2608_30963_gb300 import synth  # noqa: E402

# (workload, source layers, target layers, target lengths, source rotary_dim)
CASES = [("tiny_fp32", 4, 2, [256, 100], 0),
         ("qwen1p5b_to_gemma2b_1k", 3, 2, [64, 17], 0),
         ("llama70b_to_qwen7b_8k", 5, 3, [48], 64)]
SAMPLES = 48


def key(name, Ls, Lt, lens, rot):
    return f"{name}:{Ls}:{Lt}:{'-'.join(map(str, lens))}:{rot}"


def case_outputs(name, Ls, Lt, lens, rot):
    spec = synth.config_specs()[name]
    spec = dataclasses.replace(spec, src=dataclasses.replace(spec.src, num_layers=Ls, rotary_dim=rot),
                               dst=dataclasses.replace(spec.dst, num_layers=Lt))
    c = make_case(spec, lens)
    ok, ov = oracle_problem(c).translate()
    rng = np.random.default_rng(99)
    idx = [[int(rng.integers(0, n)) for n in ok.shape] for _ in range(SAMPLES)]
    spans = c.wl.span_lo is not None
    return {"index": idx, "k": [float(ok[tuple(i)]) for i in idx], "v": [float(ov[tuple(i)]) for i in idx],
            "layer_map": [int(x) for x in np.ravel(c.layer_map)],
            "span_lo": [int(x) for x in c.wl.span_lo[:32]] if spans else [],
            "span_hi": [int(x) for x in c.wl.span_hi[:32]] if spans else []}


def build():
    return {key(*cs): case_outputs(*cs) for cs in CASES}


if __name__ == "__main__":
    cases = build()
    with open(os.path.join(HERE, "oracle_regression.json"), "w") as f:   # one case per line
        f.write("{\n" + ",\n".join(f"{json.dumps(k)}: {json.dumps(v, separators=(',', ':'))}"
                                    for k, v in cases.items()) + "\n}\n")
