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


_NCU_CSV = """==PROF== Connected to process 1234
"ID","Process ID","Process Name","Host Name","Kernel Name","Context","Stream","Block Size","Grid Size","Device","CC","Section Name","Metric Name","Metric Unit","Metric Value"
"0","1234","python","box","void kvx::<unnamed>::translate_tc_aligned_kernel<64, 0>(kvx::<unnamed>::AlignedParams)","1","7","(608, 1, 1)","(152, 1, 1)","0","10.3","Command line profiler metrics","dram__bytes_read.sum","Mbyte","243.40"
"0","1234","python","box","void kvx::<unnamed>::translate_tc_aligned_kernel<64, 0>(kvx::<unnamed>::AlignedParams)","1","7","(608, 1, 1)","(152, 1, 1)","0","10.3","Command line profiler metrics","dram__bytes_write.sum","Kbyte","56,734.72"
"0","1234","python","box","void kvx::<unnamed>::translate_tc_aligned_kernel<64, 0>(kvx::<unnamed>::AlignedParams)","1","7","(608, 1, 1)","(152, 1, 1)","0","10.3","Command line profiler metrics","gpu__time_duration.sum","usecond","76.10"
"""


def test_traffic_record_from_an_ncu_csv_and_its_lookup(bench, tmp_path, monkeypatch):
    """record_traffic sums read and write bytes of the identity-kernel launch (units converted),
    and the bench reports them only for the same workload and unchanged kernel sources."""
    csv_path = tmp_path / "traffic.csv"
    csv_path.write_text(_NCU_CSV)
    rec_path = tmp_path / "traffic.json"
    monkeypatch.setattr(bench, "_TRAFFIC_REC", str(rec_path))
    assert bench.record_traffic(str(csv_path), "qwen7b_to_qwen1p5b_4k", "ncu ...") == 0
    import json
    rec = json.loads(rec_path.read_text())
    assert rec["dram_bytes_read"] == 243_400_000 and rec["dram_bytes_write"] == 56_734_720
    assert rec["dram_bytes_per_launch"] == 243_400_000 + 56_734_720
    assert rec["kernel"] == "translate_tc_aligned_kernel<64, 0>"
    assert abs(rec["duration_s"] - 76.10e-6) < 1e-12
    assert bench.traffic_for("qwen7b_to_qwen1p5b_4k", str(rec_path)) == rec["dram_bytes_per_launch"]
    assert bench.traffic_for("longctx_32k_b8", str(rec_path)) is None
    rec["kernel_rev"] = "0" * 12          # a capture of other sources
    rec_path.write_text(json.dumps(rec))
    assert bench.traffic_for("qwen7b_to_qwen1p5b_4k", str(rec_path)) is None


def test_traffic_record_without_the_identity_kernel_is_refused(bench, tmp_path, monkeypatch):
    csv_path = tmp_path / "traffic.csv"
    csv_path.write_text(_NCU_CSV.replace("translate_tc_aligned_kernel", "translate_tc_kernel"))
    rec_path = tmp_path / "traffic.json"
    monkeypatch.setattr(bench, "_TRAFFIC_REC", str(rec_path))
    assert bench.record_traffic(str(csv_path), "qwen7b_to_qwen1p5b_4k", "ncu ...") == 1
    assert not rec_path.exists()
