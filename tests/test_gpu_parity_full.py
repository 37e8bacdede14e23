"""Whole-output parity at full size, and the token alignments a tokenizer pair really produces.

- Every element of every full-size workload's output (in the launch configuration bench.py
  times) against the oracle, the oracle split over spawned processes by (target layer,
  sequence).  Cross-tokenizer workloads build their spans on the device from the two
  tokenisations' byte offsets first, as the bench does.
- Spans from two independent tokenisations of the same bytes (synth.draw_tokenizations),
  aligned on the device by kvx_build_alignment and fed to kvx_translate: a finer target
  (several target tokens on one source token), a coarser one (long spans), equal grains, and
  single-byte source tokens under 6-byte target tokens, whose 32-token sub-tiles need more
  source rows than the span kernel's 48-row window holds, so the global-memory gather runs on
  every full sub-tile (checked through the plan diagnostics against the plan rule).
- Non-monotone and overlapping spans, which no tokenizer pair gives but the interface allows.
"""
import dataclasses

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import paper_2608_30963_gb300 as kvx
from paper_2608_30963_gb300 import synth

import parallel_oracle
from harness import compare, explicit_span_workload, make_case, oracle_problem, tokenization_workload

pytestmark = pytest.mark.gpu
SPECS = synth.config_specs()
PATHS = [kvx.KVX_PATH_SIMT, kvx.KVX_PATH_AUTO]
WINDOW_CAP = 48   # source rows one sub-tile window of the span kernel stages


@pytest.fixture(scope="module", autouse=True)
def _lib():
    kvx.build()
    yield


def _shrink(spec, Ls, Lt, **kw):
    return dataclasses.replace(spec, src=dataclasses.replace(spec.src, num_layers=Ls),
                               dst=dataclasses.replace(spec.dst, num_layers=Lt), **kw)


# ------------------------------------------------------------------ whole output, full size
FULL_ALL = ["qwen7b_to_qwen1p5b_4k", "qwen1p5b_to_gemma2b_1k", "qwen1p5b_to_gemma2b_2k", "qwen1p5b_to_gemma2b_4k",
            "llama70b_to_qwen7b_8k", "llama70b_to_qwen7b_8k_dense", "llama70b_to_qwen7b_8k_layers2",
            "qwen7b_to_qwen1p5b_4k_latent64"]


@pytest.mark.parametrize("name", FULL_ALL)
def test_full_output_every_element(name):
    from gpu_harness import DeviceCase, i32
    spec = SPECS[name]
    c = make_case(spec)
    wl = c.wl
    g = DeviceCase(c, path=kvx.KVX_PATH_AUTO)
    if spec.cross_tokenizer:   # spans built on the device from byte offsets, as in every bench step
        lo = torch.full((wl.total_tgt,), -1, dtype=torch.int32, device="cuda")
        hi = torch.full((wl.total_tgt,), -1, dtype=torch.int32, device="cuda")
        kvx.build_alignment(i32(wl.src_seq_off), i32(wl.src_end), i32(wl.tgt_seq_off), i32(wl.tgt_end), lo, hi)
        g.span_lo, g.span_hi = lo, hi
    g.run()
    torch.cuda.synchronize()
    assert g.status() == 0
    if spec.cross_tokenizer:
        np.testing.assert_array_equal(g.span_lo.cpu().numpy(), wl.span_lo)
        np.testing.assert_array_equal(g.span_hi.cpu().numpy(), wl.span_hi)
    jobs = parallel_oracle.jobs_for(spec, wl, c.layer_map, c.src_k, c.src_v, c.w_k, c.w_v, g.gather_layer,
                                    low_rank=c.low_rank)
    parallel_oracle.check(parallel_oracle.run(jobs), f"{name}: all {len(jobs)} (layer, sequence) blocks")


# ------------------------------------------------------------------ spans from two tokenisations
def _expected_plan(wl, cap=WINDOW_CAP):
    """The span plan's window rule on the host: per 32-token sub-tile, the window starts at the
    first token's span and ends at the furthest span end of that token's sequence, cut at `cap`
    rows; tokens whose span is not inside it are gathered from global memory."""
    T = wl.total_tgt
    seq = np.searchsorted(wl.tgt_seq_off, np.arange(T), side="right") - 1
    staged = glob = subs_glob = 0
    nsub = (T + 127) // 128 * 4
    for sub in range(nsub):
        t = np.arange(sub * 32, min(sub * 32 + 32, T))
        if t.size == 0:
            continue
        lo, hi, b = wl.span_lo[t], wl.span_hi[t], seq[t]
        same = b == b[0]
        c0 = int(lo[0])
        R = min(max(int(hi[same].max()) - c0, 0), cap)
        inwin = same & (lo >= c0) & (hi <= c0 + R)
        staged += int(inwin.sum())
        glob += int((~inwin).sum())
        subs_glob += int((~inwin).any())
    return {"subtiles": nsub, "staged_tokens": staged, "global_tokens": glob, "subtiles_with_global": subs_glob}


MIXES = {"target_finer_5_2": (5.0, 2.0), "target_coarser_2_6": (2.0, 6.0), "equal_1_1": (1.0, 1.0),
         "byte_source_1_6": (1.0, 6.0)}
GEOMS = {"gemma_expansion": ("qwen1p5b_to_gemma2b_1k", 3, 2), "llama_grouped": ("llama70b_to_qwen7b_8k", 3, 2)}


@pytest.mark.parametrize("path", PATHS, ids=["simt", "auto"])
@pytest.mark.parametrize("geom", list(GEOMS))
@pytest.mark.parametrize("mix", list(MIXES))
def test_spans_from_independent_tokenizations(mix, geom, path):
    from gpu_harness import DeviceCase, i32
    base, Ls, Lt = GEOMS[geom]
    spec = _shrink(SPECS[base], Ls, Lt)
    ms, mt = MIXES[mix]
    wl = tokenization_workload(spec, [2600, 37, 1, 900], ms, mt, key=7 + list(MIXES).index(mix))
    c = make_case(spec, wl=wl)
    g = DeviceCase(c, path=path)
    lo = torch.full((wl.total_tgt,), -1, dtype=torch.int32, device="cuda")
    hi = torch.full((wl.total_tgt,), -1, dtype=torch.int32, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    kvx.build_alignment(i32(wl.src_seq_off), i32(wl.src_end), i32(wl.tgt_seq_off), i32(wl.tgt_end), lo, hi, st)
    g.span_lo, g.span_hi = lo, hi
    g.run()
    torch.cuda.synchronize()
    np.testing.assert_array_equal(lo.cpu().numpy(), wl.span_lo)   # the device builder, bit-exact
    np.testing.assert_array_equal(hi.cpu().numpy(), wl.span_hi)
    assert int(st.item()) == 0
    n = wl.span_hi - wl.span_lo
    if mix == "target_finer_5_2":
        assert (np.diff(wl.span_lo) == 0).any(), "no target tokens share a source token"
    if mix in ("target_coarser_2_6", "byte_source_1_6"):
        assert n.max() > 3
    ok, ov = oracle_problem(c).translate()
    gk, gv = g.gather()
    compare(gk, ok, "bf16", f"{mix} {geom} K")
    compare(gv, ov, "bf16", f"{mix} {geom} V")
    assert g.status() == 0
    if path == kvx.KVX_PATH_AUTO:
        stats = g.tr.span_plan_stats()
        assert stats == _expected_plan(wl), (stats, _expected_plan(wl))
        if mix == "byte_source_1_6":
            # 32 target tokens of ~6 single-byte source tokens each need ~190 rows, four times the
            # window: every sub-tile holding tokens (but at most one short one) gathers from global memory
            assert stats["subtiles_with_global"] >= (wl.total_tgt + 31) // 32 - 1, stats


@pytest.mark.parametrize("path", PATHS, ids=["simt", "auto"])
@pytest.mark.parametrize("kind", ["reversed", "random_overlapping"])
def test_non_monotone_spans(kind, path):
    from gpu_harness import DeviceCase
    spec = _shrink(SPECS["llama70b_to_qwen7b_8k"], 3, 2)
    r = np.random.default_rng(41)
    src_lens, los, his = [], [], []
    for b, T in enumerate([700, 130]):
        S = int(T * 1.3)
        if kind == "reversed":   # target token t reads the source tokens mirrored from the end
            n = r.choice([1, 2, 3], size=T, p=[0.75, 0.2, 0.05])
            lo = np.maximum(S - 1 - np.arange(T) - n + 1, 0)
            hi = np.minimum(lo + n, S)
        else:                    # any span anywhere in the sequence, of length 1..5
            n = r.integers(1, 6, size=T)
            lo = r.integers(0, S - 5, size=T)
            hi = lo + n
        src_lens.append(S); los.append(lo); his.append(hi)
    wl = explicit_span_workload(spec, src_lens, los, his)
    c = make_case(spec, wl=wl)
    g = DeviceCase(c, path=path)
    g.run()
    torch.cuda.synchronize()
    ok, ov = oracle_problem(c).translate()
    gk, gv = g.gather()
    compare(gk, ok, "bf16", f"{kind} K")
    compare(gv, ov, "bf16", f"{kind} V")
    assert g.status() == 0
    if path == kvx.KVX_PATH_AUTO:
        stats = g.tr.span_plan_stats()
        assert stats == _expected_plan(wl)
        assert stats["global_tokens"] > 0


# ------------------------------------------------------------------ long-context sweep: all nine points
LONGCTX = [f"longctx_{L}k_b{B}" for L in (8, 16, 32) for B in (1, 4, 8)]


@pytest.mark.parametrize("name", LONGCTX)
def test_longctx_sweep_device_generated(name):
    """Each point of the long-context sweep (8K/16K/32K x batch 1/4/8, varlen, paged, shuffled
    16-token pages) in the bench's launch configuration.  Inputs are drawn on the device from a
    fixed seed (host fp32 copies of the largest would need ~30 GB).  Bit-exact: paged ==
    contiguous on every layer, and the identity kernel == the span kernel (explicit identity
    spans) on three layers; every element of those three layers against the oracle."""
    from gpu_harness import i32, to_host
    spec = SPECS[name]
    wl = synth.make_workload(spec)
    s, d = spec.src, spec.dst
    gen = torch.Generator(device="cuda").manual_seed(20260 + LONGCTX.index(name))
    shape = (wl.batch, s.num_kv_heads, wl.s_max, s.head_dim)
    ks = [torch.randn(shape, generator=gen, device="cuda").to(torch.bfloat16) for _ in range(s.num_layers)]
    vs = [torch.randn(shape, generator=gen, device="cuda").to(torch.bfloat16) for _ in range(s.num_layers)]
    w_k = torch.randn((d.num_layers, d.num_kv_heads, spec.group_in, d.head_dim), generator=gen, device="cuda")
    w_v = torch.randn((d.num_layers, d.num_kv_heads, spec.group_in, d.head_dim), generator=gen, device="cuda")
    w_k = (w_k / spec.group_in ** 0.5).to(torch.bfloat16)
    w_v = (w_v / spec.group_in ** 0.5).to(torch.bfloat16)
    lm = list(range(d.num_layers))
    tr = kvx.Translator(s, d, w_k, w_v, layer_map=lm)
    src_len, seq_off = i32(wl.src_len), i32(wl.tgt_seq_off)
    T = wl.total_tgt
    pt = i32(wl.page_table)
    pool = (wl.num_pages, spec.page_size, d.num_kv_heads, d.head_dim)
    cont = (wl.batch, d.num_kv_heads, wl.t_max, d.head_dim)
    pk = [torch.full(pool, float("nan"), dtype=torch.bfloat16, device="cuda") for _ in range(d.num_layers)]
    pv = [torch.full(pool, float("nan"), dtype=torch.bfloat16, device="cuda") for _ in range(d.num_layers)]
    tr.translate(ks, vs, src_len, seq_off, T, pk, pv, page_table=pt, page_size=spec.page_size,
                 num_pages=wl.num_pages)
    assert tr.device_status() == 0
    ck = [torch.full(cont, float("nan"), dtype=torch.bfloat16, device="cuda") for _ in range(d.num_layers)]
    cv = [torch.full(cont, float("nan"), dtype=torch.bfloat16, device="cuda") for _ in range(d.num_layers)]
    tr.translate(ks, vs, src_len, seq_off, T, ck, cv)
    assert tr.device_status() == 0
    sub = [0, 13, 27]
    lo = np.concatenate([np.arange(t, dtype=np.int32) for t in wl.tgt_len])
    sk_ = [torch.full(cont, float("nan"), dtype=torch.bfloat16, device="cuda") for _ in sub]
    sv_ = [torch.full(cont, float("nan"), dtype=torch.bfloat16, device="cuda") for _ in sub]
    tr3 = kvx.Translator(s, dataclasses.replace(d, num_layers=3), w_k[sub].contiguous(), w_v[sub].contiguous(),
                         layer_map=sub)
    tr3.translate(ks, vs, src_len, seq_off, T, sk_, sv_, span_lo=i32(lo), span_hi=i32(lo + 1))
    assert tr3.device_status() == 0
    torch.cuda.synchronize()
    for b in range(wl.batch):
        n = int(wl.tgt_len[b])
        pages = torch.from_numpy(wl.page_table[b]).cuda().long()
        idx = torch.arange(n, device="cuda")
        for j in range(d.num_layers):
            for P_, C_ in ((pk[j], ck[j]), (pv[j], cv[j])):
                rows = P_[pages[idx // spec.page_size], idx % spec.page_size]       # [n, Ht, dt]
                assert torch.equal(rows.transpose(0, 1).view(torch.int16), C_[b, :, :n].view(torch.int16))
        for i, j in enumerate(sub):
            assert torch.equal(sk_[i][b, :, :n].view(torch.int16), ck[j][b, :, :n].view(torch.int16))
            assert torch.equal(sv_[i][b, :, :n].view(torch.int16), cv[j][b, :, :n].view(torch.int16))
    # every element of the three layers against the oracle
    src_k = {l: to_host(ks[l]) for l in sub}
    src_v = {l: to_host(vs[l]) for l in sub}
    spec3 = dataclasses.replace(spec, dst=dataclasses.replace(d, num_layers=3))
    wl3 = dataclasses.replace(wl, spec=spec3)

    def gpu_layer(j, kv):
        t = to_host((ck if kv == 0 else cv)[sub[j]])                           # [B, Ht, t_max, dt]
        return np.concatenate([t[b, :, :int(wl.tgt_len[b])] for b in range(wl.batch)], axis=1)

    jobs = parallel_oracle.jobs_for(spec3, wl3, sub, src_k, src_v, to_host(w_k[sub]), to_host(w_v[sub]), gpu_layer)
    parallel_oracle.check(parallel_oracle.run(jobs), f"{name}: target layers {sub}, every element")
