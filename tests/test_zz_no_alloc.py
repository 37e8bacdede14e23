"""kvx_translate_static: the allocation-free entry point.

Some callers cannot allocate device memory when they translate (a caching
allocator owns the device memory, the memory budget was fixed at start-up, or
cudaMalloc would synchronise a latency-critical path).  kvx_translate_static
serves them from a static device scratch array.  These tests call it through
the C ABI and check, on two calls in a row, that it writes what the regular
entry point (kvx_translator_create + kvx_translate) writes for the same inputs,
and that both agree with the oracle, for contiguous and paged target caches.
The file sorts last so a stop-at-first-failure run has run every other test.
"""
import dataclasses

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2608_30963_gb300 as kvx
from paper_2608_30963_gb300 import synth

from harness import compare, make_case

pytestmark = pytest.mark.gpu


def _structs(g):
    """C structs of a DeviceCase's buffers (same marshalling as Translator.translate)."""
    P = kvx._ptr
    s0 = g.src_k[0]
    src = kvx.kvx_src_kv(s0.shape[0], s0.shape[2], kvx._ptr_array(g.src_k), kvx._ptr_array(g.src_v),
                         s0.stride(0), s0.stride(1), s0.stride(2), P(g.src_len), P(g.src_pos))
    tgt = kvx.kvx_tgt_tokens(g.c.wl.total_tgt, P(g.seq_off), P(g.span_lo), P(g.span_hi), P(g.tgt_pos))
    d0 = g.dst_k[0]
    if g.paged:
        wl = g.c.wl
        dst = kvx.kvx_dst_kv(kvx._ptr_array(g.dst_k), kvx._ptr_array(g.dst_v), 1, 0, 0, 0, 0, P(g.page_table),
                             int(wl.max_pages), g.c.spec.page_size, int(wl.num_pages))
    else:
        dst = kvx.kvx_dst_kv(kvx._ptr_array(g.dst_k), kvx._ptr_array(g.dst_v), 0, d0.shape[2], d0.stride(0),
                             d0.stride(1), d0.stride(2), None, 0, 0, 0)
    return src, tgt, dst


def _shrink(spec, Ls, Lt):
    return dataclasses.replace(spec, src=dataclasses.replace(spec.src, num_layers=Ls),
                               dst=dataclasses.replace(spec.dst, num_layers=Lt))


CASES = [("tiny_fp32", None, None, None, False), ("qwen1p5b_to_gemma2b_1k", 3, 2, [130, 7], False),
         ("qwen7b_to_qwen1p5b_4k", 2, 2, [200], False), ("llama70b_to_qwen7b_8k", 3, 2, [150], False),
         ("qwen7b_to_qwen1p5b_4k_partial", 2, 2, [200], False),
         ("qwen7b_to_qwen1p5b_4k_paged", 2, 2, [200, 37], True),
         ("qwen1p5b_to_gemma2b_1k_paged", 3, 2, [130, 7], True)]


@pytest.mark.parametrize("name,Ls,Lt,lens,paged", CASES, ids=[c[0] for c in CASES])
def test_static_entry_matches_translator_on_two_calls(name, Ls, Lt, lens, paged):
    """Two calls in a row, each compared with the regular entry point on the same buffers and
    with the oracle; paged cases write through a shuffled page table."""
    from gpu_harness import DeviceCase, to_dev, i32
    from harness import oracle_problem
    kvx.build()
    name = name.removesuffix("_paged")
    spec = synth.config_specs()[name.removesuffix("_partial")]
    if Ls:
        spec = _shrink(spec, Ls, Lt)
    if name.endswith("_partial"):
        # partial rotary heads on both sides (turns of the non-rotating pairs are 0 on the device)
        spec = dataclasses.replace(spec, src=dataclasses.replace(spec.src, rotary_dim=64),
                                   dst=dataclasses.replace(spec.dst, rotary_dim=32))
    if name.startswith("llama70b"):
        # the Llama-3.1 RoPE schedule on the source side (frequencies computed on the device here)
        spec = dataclasses.replace(spec, src=dataclasses.replace(synth.LLAMA70B_SCALED, num_layers=Ls))
    c = make_case(spec, lens)
    # the regular entry point, CUDA-core path (the kernel the static entry point runs)
    ref = DeviceCase(c, path=kvx.KVX_PATH_SIMT, paged=paged)
    ref.run()
    torch.cuda.synchronize()
    rk, rv = ref.gather()
    assert ref.status() == 0
    ok, ov = oracle_problem(c).translate()

    g = DeviceCase(c, path=kvx.KVX_PATH_SIMT, paged=paged)   # buffers only; its translator is not used
    wk, wv = to_dev(c.w_k, spec.dtype), to_dev(c.w_v, spec.dtype)
    desc = g.tr.desc
    stream = torch.cuda.current_stream().cuda_stream
    for call in range(2):
        for t in g.dst_k + g.dst_v:
            t.fill_(float("nan"))
        src, tgt, dst = _structs(g)
        bits = kvx.kvx_translate_static(desc, wk.data_ptr(), wv.data_ptr(), src, tgt, dst, stream,
                                        read_status=True)
        assert bits == 0, f"call {call}: status 0x{bits:x}"
        gk, gv = g.gather()
        compare(gk, rk, spec.dtype)
        compare(gv, rv, spec.dtype)
        sk, sv = compare(gk, ok, spec.dtype), compare(gv, ov, spec.dtype)
        print(f"{name} call {call}: vs oracle K rel_l2={sk['rel_l2']:.2e} max_abs={sk['max_abs']:.3e} "
              f"n>3e-2={sk['n_above_3e-2']}; V rel_l2={sv['rel_l2']:.2e} max_abs={sv['max_abs']:.3e} "
              f"n>3e-2={sv['n_above_3e-2']}")


def test_static_entry_clears_its_status_and_rejects_oversize():
    from gpu_harness import DeviceCase, to_dev, i32
    kvx.build()
    spec = _shrink(synth.config_specs()["qwen7b_to_qwen1p5b_4k"], 2, 2)
    c = make_case(spec, [64])
    g = DeviceCase(c, path=kvx.KVX_PATH_SIMT, paged=False)
    wk, wv = to_dev(c.w_k, spec.dtype), to_dev(c.w_v, spec.dtype)
    stream = torch.cuda.current_stream().cuda_stream
    lo = np.arange(64, dtype=np.int32)
    hi = lo + 1
    hi[3] = 10_000                                   # past the source: clamped and flagged
    g.span_lo, g.span_hi = i32(lo), i32(hi)
    src, tgt, dst = _structs(g)
    bits = kvx.kvx_translate_static(g.tr.desc, wk.data_ptr(), wv.data_ptr(), src, tgt, dst, stream, True)
    assert bits & kvx.KVX_DEV_SPAN_CLAMPED
    g.span_lo = g.span_hi = None                     # a clean call right after: the word starts at zero
    src, tgt, dst = _structs(g)
    assert kvx.kvx_translate_static(g.tr.desc, wk.data_ptr(), wv.data_ptr(), src, tgt, dst, stream, True) == 0
    # weights larger than the static scratch are refused before anything runs
    big = kvx.kvx_translator_desc.from_buffer_copy(g.tr.desc)
    big.layer_map = None
    big.dst.num_layers = 128                         # 2 * 128 * 2 * 256 * 128 * 2 B > 8 MiB
    with pytest.raises(kvx.KvxError) as e:
        kvx.kvx_translate_static(big, wk.data_ptr(), wv.data_ptr(), src, tgt, dst, stream, True)
    assert e.value.status == kvx.KVX_ERR_UNSUPPORTED
