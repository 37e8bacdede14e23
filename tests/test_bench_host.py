"""bench.py's host-side arithmetic (no GPU): the roofline numerator and its layer map.

The algorithmic bytes of one translation are the distinct mapped source layers' K and V rows
read once, the target K and V rows written once and the translator weights; for the 7B->1.5B
shapes at 4K that is 28*4*4096*128*2*2 + 28*2*4096*128*2*2 + 2*28*2*256*128*2 bytes, with
2*4096*256*128*28*2*2 FLOPs.
"""
import importlib.util
import os

import numpy as np
import pytest

import oracle
from paper_2608_30963_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def bench():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_headline_bytes_and_flops(bench):
    spec = synth.config_specs()["qwen7b_to_qwen1p5b_4k"]
    wl = synth.make_workload(spec)
    a = bench.algorithmic(spec, wl, oracle.layer_map_nearest(28, 28))
    assert a["read"] == 28 * 4 * 4096 * 128 * 2 * 2 == 234_881_024
    assert a["write"] == 28 * 2 * 4096 * 128 * 2 * 2 == 117_440_512
    assert a["weights"] == 2 * 28 * 2 * 256 * 128 * 2 == 7_340_032
    assert a["bytes"] == 359_661_568
    assert a["flops"] == 2 * 4096 * 256 * 128 * 28 * 2 * 2


def test_cross_tokenizer_bytes_count_each_distinct_source_layer_once(bench):
    spec = synth.config_specs()["llama70b_to_qwen7b_8k"]
    wl = synth.make_workload(spec)
    lm = oracle.layer_map_nearest(80, 28)
    a = bench.algorithmic(spec, wl, lm)
    S = int(wl.src_len.sum())
    assert a["read"] == len(set(lm.tolist())) * 8 * S * 128 * 2 * 2
    assert a["write"] == 28 * 4 * wl.total_tgt * 128 * 2 * 2
    # a latent adapter counts its two factors, not the folded matrix
    lat = synth.config_specs()["qwen7b_to_qwen1p5b_4k_latent64"]
    b = bench.algorithmic(lat, synth.make_workload(lat), oracle.layer_map_nearest(28, 28))
    assert b["weights"] == 2 * 28 * 2 * 64 * (256 + 128) * 2


@pytest.mark.parametrize("Ls,Lt", [(28, 28), (80, 28), (28, 26), (4, 2), (3, 5), (7, 1), (1, 1), (2, 9)])
def test_bench_layer_map_equals_the_oracle(bench, Ls, Lt):
    assert bench.nearest_map(Ls, Lt) == [int(x) for x in oracle.layer_map_nearest(Ls, Lt)]
