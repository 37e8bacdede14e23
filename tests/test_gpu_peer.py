"""kvx_translate_to_device: the translated cache written into the target model's GPU.

On one GPU the "remote" target cache is a separate allocation on the same device: both modes
(kernel stores, staged copy) must give the oracle's result and the same bits as kvx_translate.
The two-GPU case (source on device 0, target cache on device 1) runs only where the process
sees two devices.
"""
import dataclasses

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2608_30963_gb300 as kvx
from paper_2608_30963_gb300 import synth

from harness import compare, make_case, oracle_problem

pytestmark = pytest.mark.gpu
SPECS = synth.config_specs()


@pytest.fixture(scope="module", autouse=True)
def _lib():
    kvx.build()
    yield


def _shrink(spec, Ls, Lt):
    return dataclasses.replace(spec, src=dataclasses.replace(spec.src, num_layers=Ls),
                               dst=dataclasses.replace(spec.dst, num_layers=Lt))


CASES = {"identity_tma": ("qwen7b_to_qwen1p5b_4k", 3, 2, [300, 129], kvx.KVX_PATH_AUTO),
         "spans_expansion": ("qwen1p5b_to_gemma2b_1k", 3, 2, [300, 41], kvx.KVX_PATH_AUTO),
         "spans_grouped_simt": ("llama70b_to_qwen7b_8k", 3, 2, [200], kvx.KVX_PATH_SIMT)}


def _like(ts, device):
    return [torch.full(t.shape, float("nan"), dtype=t.dtype, device=device) for t in ts]


@pytest.mark.parametrize("paged", [False, True], ids=["contiguous", "paged"])
@pytest.mark.parametrize("mode", [kvx.KVX_PEER_STORES, kvx.KVX_PEER_STAGED], ids=["stores", "staged"])
@pytest.mark.parametrize("name", list(CASES))
def test_translate_into_another_cache_on_one_device(name, mode, paged):
    from gpu_harness import DeviceCase
    base, Ls, Lt, lens, path = CASES[name]
    c = make_case(_shrink(SPECS[base], Ls, Lt), lens)
    g = DeviceCase(c, path=path, paged=paged)
    g.run()                                          # kvx_translate into g's own target cache
    torch.cuda.synchronize()
    ref_k, ref_v = g.gather()
    wl = c.wl
    dev = torch.cuda.current_device()
    out_k, out_v = _like(g.dst_k, dev), _like(g.dst_v, dev)
    kw = dict(span_lo=g.span_lo, span_hi=g.span_hi, page_table=g.page_table, page_size=c.spec.page_size,
              num_pages=wl.num_pages if g.paged else 0)
    if mode == kvx.KVX_PEER_STAGED and paged:
        with pytest.raises(kvx.KvxError) as e:
            g.tr.translate_to_device(g.src_k, g.src_v, g.src_len, g.seq_off, wl.total_tgt, out_k, out_v, dev, mode,
                                     staging_k=_like(g.dst_k, dev), staging_v=_like(g.dst_v, dev), **kw)
        assert e.value.status == kvx.KVX_ERR_UNSUPPORTED
        return
    stg = {}
    if mode == kvx.KVX_PEER_STAGED:
        stg = dict(staging_k=_like(g.dst_k, dev), staging_v=_like(g.dst_v, dev))
    g.tr.translate_to_device(g.src_k, g.src_v, g.src_len, g.seq_off, wl.total_tgt, out_k, out_v, dev, mode,
                             **stg, **kw)
    torch.cuda.synchronize()
    assert g.status() == 0
    g.dst_k, g.dst_v = out_k, out_v
    gk, gv = g.gather()
    np.testing.assert_array_equal(gk.view(np.uint32), ref_k.view(np.uint32))   # the same bits as kvx_translate
    np.testing.assert_array_equal(gv.view(np.uint32), ref_v.view(np.uint32))
    ok, ov = oracle_problem(c).translate()
    compare(gk, ok, "bf16", f"{name} mode {mode} K")
    compare(gv, ov, "bf16", f"{name} mode {mode} V")


def test_staged_mode_argument_checks():
    from gpu_harness import DeviceCase
    c = make_case(_shrink(SPECS["qwen7b_to_qwen1p5b_4k"], 2, 2), [64])
    g = DeviceCase(c, paged=False)
    wl = c.wl
    dev = torch.cuda.current_device()
    out_k, out_v = _like(g.dst_k, dev), _like(g.dst_v, dev)
    with pytest.raises(kvx.KvxError) as e:   # no staging cache
        g.tr.translate_to_device(g.src_k, g.src_v, g.src_len, g.seq_off, wl.total_tgt, out_k, out_v, dev,
                                 kvx.KVX_PEER_STAGED)
    assert e.value.status == kvx.KVX_ERR_INVALID_ARG
    with pytest.raises(kvx.KvxError) as e:   # target memory on another device than named
        g.tr.translate_to_device(g.src_k, g.src_v, g.src_len, g.seq_off, wl.total_tgt, out_k, out_v, dev + 1,
                                 kvx.KVX_PEER_STORES)
    assert e.value.status == kvx.KVX_ERR_INVALID_ARG
    small = [t[:, :, :32].contiguous() for t in g.dst_k]   # staging of another layout
    with pytest.raises(kvx.KvxError) as e:
        g.tr.translate_to_device(g.src_k, g.src_v, g.src_len, g.seq_off, wl.total_tgt, out_k, out_v, dev,
                                 kvx.KVX_PEER_STAGED, staging_k=small, staging_v=small)
    assert e.value.status == kvx.KVX_ERR_INVALID_ARG
    kvx.kvx_enable_peer(dev)                 # the current device itself: accepted, nothing to do


@pytest.mark.skipif(not torch.cuda.is_available() or torch.cuda.device_count() < 2,
                    reason="needs two GPUs in the process")
@pytest.mark.parametrize("mode", [kvx.KVX_PEER_STORES, kvx.KVX_PEER_STAGED], ids=["stores", "staged"])
def test_translate_into_a_second_gpu(mode):
    """Source caches and translator on device 0, target cache on device 1."""
    from gpu_harness import DeviceCase
    torch.cuda.set_device(0)
    c = make_case(_shrink(SPECS["qwen1p5b_to_gemma2b_1k"], 3, 2), [300, 41])
    g = DeviceCase(c, paged=False)
    wl = c.wl
    kvx.kvx_enable_peer(1)
    out_k, out_v = _like(g.dst_k, 1), _like(g.dst_v, 1)
    stg = dict(staging_k=_like(g.dst_k, 0), staging_v=_like(g.dst_v, 0)) if mode == kvx.KVX_PEER_STAGED else {}
    g.tr.translate_to_device(g.src_k, g.src_v, g.src_len, g.seq_off, wl.total_tgt, out_k, out_v, 1, mode,
                             span_lo=g.span_lo, span_hi=g.span_hi, **stg)
    torch.cuda.synchronize(0)
    torch.cuda.synchronize(1)
    assert g.status() == 0
    g.dst_k, g.dst_v = [t.to(0) for t in out_k], [t.to(0) for t in out_v]
    gk, gv = g.gather()
    ok, ov = oracle_problem(c).translate()
    compare(gk, ok, "bf16", f"two GPUs mode {mode} K")
    compare(gv, ov, "bf16", f"two GPUs mode {mode} V")
