"""CUDA path vs the CPU oracle, through the C ABI, on seeded synthetic inputs.

Small cases are compared element by element over the whole output (several
128-token tiles plus a ragged tail).  Full-size workloads, in the launch
configuration bench.py times, are compared on sampled rows the oracle computes
one by one.  Integer outputs (alignment spans) must be bit-exact.
"""
import dataclasses

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle
import paper_2608_30963_gb300 as kvx
from paper_2608_30963_gb300 import synth

from harness import compare, make_case, oracle_problem, sample_rows

pytestmark = pytest.mark.gpu

SPECS = synth.config_specs()
PATHS = [kvx.KVX_PATH_SIMT, kvx.KVX_PATH_AUTO]


@pytest.fixture(scope="module", autouse=True)
def _lib():
    kvx.build()
    yield


def _run(c, path, paged=None, max_position=0):
    from gpu_harness import DeviceCase
    g = DeviceCase(c, path=path, paged=paged, max_position=max_position)
    g.run()
    torch.cuda.synchronize()
    return g


def _full_compare(c, path, paged=None, max_position=0):
    g = _run(c, path, paged, max_position)
    ok, ov = oracle_problem(c).translate()
    gk, gv = g.gather()
    sk = compare(gk, ok, c.spec.dtype)
    sv = compare(gv, ov, c.spec.dtype)
    assert g.status() == 0
    return g, sk, sv


def _shrink(spec, Ls, Lt, **kw):
    return dataclasses.replace(spec, src=dataclasses.replace(spec.src, num_layers=Ls),
                               dst=dataclasses.replace(spec.dst, num_layers=Lt), **kw)


# ------------------------------------------------------------------ small, whole output
def test_tiny_fp32_full():
    c = make_case(SPECS["tiny_fp32"])
    _, sk, sv = _full_compare(c, kvx.KVX_PATH_AUTO)
    assert sk["max_abs"] < 1e-4 and sv["max_abs"] < 1e-4


SMALL = {
    # name: (base spec, Ls, Lt, target lengths)
    "qwen7b_qwen1p5b": ("qwen7b_to_qwen1p5b_4k", 3, 3, [300]),
    "qwen1p5b_gemma2b": ("qwen1p5b_to_gemma2b_1k", 4, 3, [300]),
    "llama70b_qwen7b": ("llama70b_to_qwen7b_8k", 9, 4, [300]),
    "longctx_paged_varlen": ("longctx_8k_b4", 2, 2, [37, 300, 129, 1]),
}


@pytest.mark.parametrize("path", PATHS, ids=["simt", "auto"])
@pytest.mark.parametrize("name", list(SMALL))
def test_small_full_output(name, path):
    base, Ls, Lt, lens = SMALL[name]
    spec = _shrink(SPECS[base], Ls, Lt)
    c = make_case(spec, lens, pad_value=float("nan"))
    _full_compare(c, path)


@pytest.mark.parametrize("path", PATHS, ids=["simt", "auto"])
def test_explicit_positions_and_layer_map(path):
    spec = _shrink(SPECS["llama70b_to_qwen7b_8k"], 5, 3, layer_map=[4, 0, 2])
    wl = synth.make_workload(spec, [200, 77])
    rng = np.random.default_rng(3)
    src_pos = rng.integers(0, 120000, size=(wl.batch, wl.s_max)).astype(np.int32)
    tgt_pos = (np.arange(wl.total_tgt) * 7 + 3000).astype(np.int32)
    c = make_case(spec, [200, 77], src_pos=src_pos, tgt_pos=tgt_pos)
    _full_compare(c, path, max_position=1 << 17)


LINEAR4 = dict(rope_type=synth.ROPE_LINEAR, rope_factor=4.0)
SCHEDULES = {
    # Llama-3.1 scaled source RoPE, cross-tokenizer (span kernel)
    "llama3_src_spans": ("llama70b_to_qwen7b_8k", 5, 3, [300, 41], dict(src=synth.LLAMA70B_SCALED), {}),
    # linear target schedule, identity alignment: source and target rotations differ
    "linear_dst_identity": ("qwen7b_to_qwen1p5b_4k", 2, 2, [300, 5], {}, LINEAR4),
    # the same scaled schedule on both sides: source and target rotations coincide
    "llama3_both_identity": ("qwen7b_to_qwen1p5b_4k", 2, 2, [300],
                             dict(rope_type=synth.ROPE_LLAMA3, rope_factor=8.0, rope_low_freq_factor=1.0,
                                  rope_high_freq_factor=4.0, rope_original_max_position=256),
                             dict(rope_type=synth.ROPE_LLAMA3, rope_factor=8.0, rope_low_freq_factor=1.0,
                                  rope_high_freq_factor=4.0, rope_original_max_position=256)),
}


@pytest.mark.parametrize("path", PATHS, ids=["simt", "auto"])
@pytest.mark.parametrize("name", list(SCHEDULES))
def test_rope_schedules(name, path):
    base, Ls, Lt, lens, src_kw, dst_kw = SCHEDULES[name]
    spec = _shrink(SPECS[base], Ls, Lt)
    src = src_kw.get("src", dataclasses.replace(spec.src, **{k: v for k, v in src_kw.items() if k != "src"}))
    src = dataclasses.replace(src, num_layers=Ls)
    spec = dataclasses.replace(spec, src=src, dst=dataclasses.replace(spec.dst, **dst_kw))
    c = make_case(spec, lens, pad_value=float("nan"))
    _full_compare(c, path)


PARTIAL = {
    # (base, Ls, Lt, target lengths, source rotary_dim, target geometry changes); identity
    # alignment with a partial rotary head runs on the span kernel (the identity kernel
    # rotates whole heads only)
    # same partial head on both sides
    "both64_identity": ("qwen7b_to_qwen1p5b_4k", 2, 2, [300, 5], 64, dict(rotary_dim=64)),
    # a quarter of the source head rotates, the target head fully: source side only
    "src32_identity": ("qwen7b_to_qwen1p5b_4k", 2, 2, [300], 32, {}),
    # d_t = 256 in two output tiles, 96 rotating channels: row stores split in up to four runs
    "dst96_identity_split": ("qwen7b_to_qwen1p5b_4k", 2, 2, [300, 41], 0,
                             dict(head_dim=256, rope_base=1e4, rotary_dim=96)),
    # cross-tokenizer spans: partial source (lanes past rhalf do not rotate), partial target
    "src64_spans": ("llama70b_to_qwen7b_8k", 5, 3, [300, 41], 64, {}),
    "dst128_spans_gemma": ("qwen1p5b_to_gemma2b_1k", 3, 2, [300], 0, dict(rotary_dim=128)),
    # fp32 caches: the CUDA-core kernel
    "both32_tiny_fp32": ("tiny_fp32", 4, 2, [256, 100], 32, dict(rotary_dim=32)),
}


@pytest.mark.parametrize("path", PATHS, ids=["simt", "auto"])
@pytest.mark.parametrize("name", list(PARTIAL))
def test_partial_rotary_heads(name, path):
    base, Ls, Lt, lens, rot_s, dst_kw = PARTIAL[name]
    spec = _shrink(SPECS[base], Ls, Lt)
    spec = dataclasses.replace(spec, src=dataclasses.replace(spec.src, rotary_dim=rot_s),
                               dst=dataclasses.replace(spec.dst, **dst_kw))
    c = make_case(spec, lens, pad_value=float("nan"))
    g, _, _ = _full_compare(c, path)
    if path == kvx.KVX_PATH_AUTO and spec.dtype == "bf16":
        assert g.tr.info().path == kvx.KVX_PATH_TCGEN05


FORMS = {
    # one map per target layer over all 8 source heads: in = 1024, streamed weight pieces
    "dense_in1024_spans": ("llama70b_to_qwen7b_8k_dense", 5, 3, [300, 41], {}),
    # dense over 2 source heads (in = 256, resident weights), expansion-shaped geometry, spans
    "dense_in256_spans": ("qwen1p5b_to_gemma2b_1k", 3, 2, [300], dict(form=synth.FORM_DENSE)),
    # dense in = 256 with identity alignment (tensor-TMA kernel)
    "dense_in256_identity": ("qwen7b_to_qwen1p5b_4k", 2, 2, [300, 5],
                             dict(form=synth.FORM_DENSE, src=synth.QWEN1P5B)),
    # groups of two source layers: in = 512, streamed weight pieces
    "layers2_in512_spans": ("llama70b_to_qwen7b_8k_layers2", 5, 3, [300, 41],
                            dict(layer_map=[[0, 1], [2, 3], [4, 4]])),
    # latent adapters, identity alignment and spans
    "latent64_identity": ("qwen7b_to_qwen1p5b_4k_latent64", 2, 2, [300, 5], {}),
    "latent16_spans": ("llama70b_to_qwen7b_8k", 5, 3, [300], dict(rank=16)),
}


@pytest.mark.parametrize("path", PATHS, ids=["simt", "auto"])
@pytest.mark.parametrize("name", list(FORMS))
def test_translator_forms(name, path):
    base, Ls, Lt, lens, kw = FORMS[name]
    spec = _shrink(SPECS[base], Ls, Lt)
    kw = dict(kw)
    if "src" in kw:
        kw["src"] = dataclasses.replace(kw["src"], num_layers=Ls)
    spec = dataclasses.replace(spec, **kw)
    c = make_case(spec, lens, pad_value=float("nan"))
    g, _, _ = _full_compare(c, path)
    if path == kvx.KVX_PATH_AUTO:
        assert g.tr.info().path == kvx.KVX_PATH_TCGEN05


HEAD_DIMS = {
    # source / target head dims other than 128: every instantiation of the tensor-core kernels
    "ds64_dt64": (synth.ModelGeom(2, 4, 64, 1e4), synth.ModelGeom(2, 2, 64, 1e4)),
    "ds256_dt128": (synth.ModelGeom(2, 2, 256, 1e4), synth.ModelGeom(2, 2, 128, 1e6)),
    "ds256_dt256_expand": (synth.ModelGeom(2, 1, 256, 1e6), synth.ModelGeom(2, 2, 256, 1e4)),
    "ds64_dt256": (synth.ModelGeom(3, 4, 64, 1e6), synth.ModelGeom(2, 1, 256, 1e4)),
}


@pytest.mark.parametrize("path", PATHS, ids=["simt", "auto"])
@pytest.mark.parametrize("spans", [False, True], ids=["identity", "spans"])
@pytest.mark.parametrize("name", list(HEAD_DIMS))
def test_head_dims(name, spans, path):
    src, dst = HEAD_DIMS[name]
    spec = synth.WorkloadSpec(name, src, dst, "bf16", [300], spans, None, True)
    c = make_case(spec, [300, 77], pad_value=float("nan"))
    g, _, _ = _full_compare(c, path)
    if path == kvx.KVX_PATH_AUTO:
        assert g.tr.info().path == kvx.KVX_PATH_TCGEN05


def test_tiny_token_counts_and_empty_sequences():
    spec = _shrink(SPECS["qwen1p5b_to_gemma2b_1k"], 2, 2)
    c = make_case(spec, [1, 0, 2, 0, 129])
    for path in PATHS:
        _full_compare(c, path)


# ------------------------------------------------------------------ invariances (bit-exact)
@pytest.mark.parametrize("path", PATHS, ids=["simt", "auto"])
def test_paged_equals_contiguous_and_batch_invariance(path):
    spec = _shrink(SPECS["longctx_8k_b4"], 2, 2)
    c = make_case(spec, [37, 300, 129])
    gp = _run(c, path, paged=True)
    gc = _run(c, path, paged=False)
    pk, pv = gp.gather()
    ck, cv = gc.gather()
    np.testing.assert_array_equal(pk, ck)
    np.testing.assert_array_equal(pv, cv)
    solo = make_case(spec, [300])
    # the second sequence alone: same source rows, same weights
    for l in solo.src_k:
        solo.src_k[l] = c.src_k[l][1:2, :, :300]
        solo.src_v[l] = c.src_v[l][1:2, :, :300]
    gs = _run(solo, path, paged=False)
    sk, sv = gs.gather()
    np.testing.assert_array_equal(sk, ck[:, :, 37:337])
    np.testing.assert_array_equal(sv, cv[:, :, 37:337])


# ------------------------------------------------------------------ full-size, sampled rows
FULL = ["qwen7b_to_qwen1p5b_4k", "qwen1p5b_to_gemma2b_1k", "qwen1p5b_to_gemma2b_2k", "qwen1p5b_to_gemma2b_4k",
        "llama70b_to_qwen7b_8k", "longctx_8k_b4", "tiny_fp32", "llama70b_to_qwen7b_8k_dense",
        "qwen7b_to_qwen1p5b_4k_latent64"]


def test_layer_groups_8k_sampled():
    """Groups of two source layers at the full 8K context, on 6 target layers (the full
    28-layer map would hold 56 source layers in host memory)."""
    spec = dataclasses.replace(SPECS["llama70b_to_qwen7b_8k_layers2"],
                               dst=dataclasses.replace(SPECS["llama70b_to_qwen7b_8k_layers2"].dst, num_layers=6),
                               layer_map=synth.layer_groups(80, 6, 2))
    c = make_case(spec)
    g = _run(c, kvx.KVX_PATH_AUTO)
    p = oracle_problem(c)
    rows = sample_rows(c, 300)
    compare(np.stack([g.row(*r) for r in rows]), np.stack([p.row(*r) for r in rows]), "bf16")
    assert g.status() == 0


@pytest.mark.parametrize("name", FULL)
def test_full_size_sampled(name):
    c = make_case(SPECS[name])
    g = _run(c, kvx.KVX_PATH_AUTO)
    p = oracle_problem(c)
    rows = sample_rows(c, 400)
    gpu = np.stack([g.row(*r) for r in rows])
    ref = np.stack([p.row(*r) for r in rows])
    compare(gpu, ref, c.spec.dtype)
    assert g.status() == 0


# ------------------------------------------------------------------ alignment builder
@pytest.mark.parametrize("key,ms,mt", [(0, 4.0, 4.0), (1, 5.0, 2.0), (2, 2.0, 6.0), (3, 1.0, 1.0)])
def test_alignment_builder_bit_exact(key, ms, mt):
    from gpu_harness import i32
    src_ends, tgt_ends = [], []
    for i, nb in enumerate([1, 57, 5000, 911]):
        se, te = synth.draw_tokenizations(nb, ms, mt, key * 10 + i)
        src_ends.append(se); tgt_ends.append(te)
    so = np.concatenate([[0], np.cumsum([len(x) for x in src_ends])]).astype(np.int32)
    to = np.concatenate([[0], np.cumsum([len(x) for x in tgt_ends])]).astype(np.int32)
    se, te = np.concatenate(src_ends), np.concatenate(tgt_ends)
    lo_ref, hi_ref, n = oracle.build_alignment(so, se, to, te)
    T = int(to[-1])
    lo = torch.full((T,), -7, dtype=torch.int32, device="cuda")
    hi = torch.full((T,), -7, dtype=torch.int32, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    kvx.build_alignment(i32(so), i32(se), i32(to), i32(te), lo, hi, st)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(lo.cpu().numpy(), lo_ref)
    np.testing.assert_array_equal(hi.cpu().numpy(), hi_ref)
    assert int(st.item()) == 0 and n == 0


def test_alignment_builder_recovers_generated_spans():
    from gpu_harness import i32
    spec = SPECS["qwen1p5b_to_gemma2b_4k"]
    wl = synth.make_workload(spec, [4096, 1000, 3])
    T = wl.total_tgt
    lo = torch.empty(T, dtype=torch.int32, device="cuda")
    hi = torch.empty(T, dtype=torch.int32, device="cuda")
    kvx.build_alignment(i32(wl.src_seq_off), i32(wl.src_end), i32(wl.tgt_seq_off), i32(wl.tgt_end), lo, hi)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(lo.cpu().numpy(), wl.span_lo)
    np.testing.assert_array_equal(hi.cpu().numpy(), wl.span_hi)


# ------------------------------------------------------------------ device status (no faults)
@pytest.mark.parametrize("path", PATHS, ids=["simt", "auto"])
def test_bad_spans_pages_positions_set_status_bits(path):
    from gpu_harness import DeviceCase, i32
    spec = _shrink(SPECS["longctx_8k_b4"], 2, 2)
    c = make_case(spec, [40, 20])
    g = DeviceCase(c, path=path, paged=True)
    T = c.wl.total_tgt
    lo = np.arange(T, dtype=np.int32) - np.repeat(c.wl.tgt_seq_off[:-1], c.wl.tgt_len)
    hi = lo + 1
    hi[5] = 10_000          # past the source length
    g.span_lo, g.span_hi = i32(lo), i32(hi)
    g.run()
    assert g.status() & kvx.KVX_DEV_SPAN_CLAMPED
    g.span_lo = g.span_hi = None
    pt = c.wl.page_table.copy()
    pt[1, 0] = 10_000       # page outside the pool
    g.page_table = i32(pt)
    g.run()
    assert g.status() == kvx.KVX_DEV_PAGE_INVALID
    g.page_table = i32(c.wl.page_table)
    g.tgt_pos = i32(np.full(T, 1 << 30, np.int32))
    g.run()
    assert g.status() == kvx.KVX_DEV_POS_CLAMPED
    g.tgt_pos = None
    g.run()
    assert g.status() == 0


def test_invalid_arguments_rejected_before_launch():
    from gpu_harness import DeviceCase
    spec = _shrink(SPECS["qwen7b_to_qwen1p5b_4k"], 2, 2)
    c = make_case(spec, [64])
    g = DeviceCase(c)
    g.span_hi = None          # span_lo without span_hi
    g.span_lo = g.seq_off
    with pytest.raises(kvx.KvxError) as e:
        g.run()
    assert e.value.status == kvx.KVX_ERR_INVALID_ARG
    bad = synth.ModelGeom(2, 3, 128, 1e6)
    with pytest.raises(kvx.KvxError) as e:
        kvx.Translator(bad, spec.dst, torch.zeros(1, device="cuda"), torch.zeros(1, device="cuda"))
    assert e.value.status == kvx.KVX_ERR_UNSUPPORTED


# ------------------------------------------------------------------ the two tensor-core kernels agree
@pytest.mark.parametrize("base,Ls,Lt,lens", [("qwen7b_to_qwen1p5b_4k", 2, 2, [300, 5, 129]),
                                             ("qwen1p5b_to_gemma2b_1k", 2, 2, [300]),
                                             ("llama70b_to_qwen7b_8k", 3, 2, [257])])
def test_identity_kernel_equals_span_kernel(base, Ls, Lt, lens):
    """Identity alignment (no span arrays) runs the tensor-TMA kernel; the same
    spans given explicitly run the span-gather kernel.  Same arithmetic: equal bits."""
    from gpu_harness import i32
    spec = _shrink(SPECS[base], Ls, Lt, cross_tokenizer=False)
    c = make_case(spec, lens)
    ga = _run(c, kvx.KVX_PATH_AUTO)
    from gpu_harness import DeviceCase
    gs = DeviceCase(c, path=kvx.KVX_PATH_AUTO)
    lo = np.concatenate([np.arange(t, dtype=np.int32) for t in lens])
    gs.span_lo, gs.span_hi = i32(lo), i32(lo + 1)
    gs.run()
    torch.cuda.synchronize()
    ak, av = ga.gather()
    sk, sv = gs.gather()
    np.testing.assert_array_equal(ak, sk)
    np.testing.assert_array_equal(av, sv)
    assert ga.status() == 0 and gs.status() == 0


# ------------------------------------------------------------------ largest workload: properties + sampled rows
def test_longctx_32k_b8_device_generated():
    """The 32K x 8 paged workload (~196K target tokens).  Inputs are drawn on the device
    from a fixed seed (host fp32 copies would need ~30 GB).  Checks, bit-exact: paged ==
    contiguous and identity kernel == span kernel (explicit identity spans); and sampled
    rows against the oracle, which reads the sampled layers copied back to the host."""
    from gpu_harness import i32, to_host
    spec = SPECS["longctx_32k_b8"]
    wl = synth.make_workload(spec)
    s, d = spec.src, spec.dst
    gen = torch.Generator(device="cuda").manual_seed(20260)
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
    lo = np.concatenate([np.arange(t, dtype=np.int32) for t in wl.tgt_len])
    sk_ = [torch.full(cont, float("nan"), dtype=torch.bfloat16, device="cuda") for _ in range(3)]
    sv_ = [torch.full(cont, float("nan"), dtype=torch.bfloat16, device="cuda") for _ in range(3)]
    # span kernel on three layers (a 3-layer translator over the same source layers 0, 13, 27)
    sub = [0, 13, 27]
    tr3 = kvx.Translator(s, dataclasses.replace(d, num_layers=3), w_k[sub].contiguous(), w_v[sub].contiguous(),
                         layer_map=sub)
    tr3.translate(ks, vs, src_len, seq_off, T, sk_, sv_, span_lo=i32(lo), span_hi=i32(lo + 1))
    assert tr3.device_status() == 0
    torch.cuda.synchronize()
    for b in range(wl.batch):
        n = int(wl.tgt_len[b])
        pages = torch.from_numpy(wl.page_table[b]).cuda().long()
        for j in range(d.num_layers):
            for P_, C_ in ((pk[j], ck[j]), (pv[j], cv[j])):
                idx = torch.arange(n, device="cuda")
                rows = P_[pages[idx // spec.page_size], idx % spec.page_size]       # [n, Ht, dt]
                assert torch.equal(rows.transpose(0, 1).view(torch.int16), C_[b, :, :n].view(torch.int16))
        for i, j in enumerate(sub):
            assert torch.equal(sk_[i][b, :, :n].view(torch.int16), ck[j][b, :, :n].view(torch.int16))
            assert torch.equal(sv_[i][b, :, :n].view(torch.int16), cv[j][b, :, :n].view(torch.int16))
    # sampled rows against the oracle on the three layers
    src_k = {l: to_host(ks[l]) for l in sub}
    src_v = {l: to_host(vs[l]) for l in sub}
    dummy = src_k[0]
    p = oracle.OracleProblem(s, dataclasses.replace(d, num_layers=3), [0, 13, 27], wl.src_len, wl.tgt_seq_off,
                             wl.s_max, wl.t_max, [src_k.get(l, dummy) for l in range(s.num_layers)],
                             [src_v.get(l, dummy) for l in range(s.num_layers)],
                             to_host(w_k[sub]), to_host(w_v[sub]))
    r = np.random.default_rng(5)
    gpu, ref = [], []
    for _ in range(300):
        i, h, kv = int(r.integers(3)), int(r.integers(d.num_kv_heads)), int(r.integers(2))
        tp = int(r.integers(T))
        b = int(np.searchsorted(wl.tgt_seq_off, tp, side="right") - 1)
        t = tp - int(wl.tgt_seq_off[b])
        gpu.append(to_host((ck if kv == 0 else cv)[sub[i]][b, h, t]))
        ref.append(p.row(i, h, kv, tp))
    compare(np.stack(gpu), np.stack(ref), "bf16")


# ------------------------------------------------------------------ graphs and streams
@pytest.mark.parametrize("base,lens", [("qwen7b_to_qwen1p5b_4k", [300, 129]), ("qwen1p5b_to_gemma2b_1k", [300])])
def test_translate_captured_in_a_cuda_graph_equals_eager(base, lens):
    """kvx_translate allocates nothing and never synchronises: captured in a CUDA graph and
    replayed twice, it writes the same bits as an eager call."""
    spec = _shrink(SPECS[base], 2, 2)
    c = make_case(spec, lens)
    g = _run(c, kvx.KVX_PATH_AUTO)
    ek, ev = g.gather()
    for t in g.dst_k + g.dst_v:
        t.fill_(float("nan"))
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(s):
        g.run(stream=s)          # warm-up on the capture stream
        s.synchronize()
        for t in g.dst_k + g.dst_v:
            t.fill_(float("nan"))
        with torch.cuda.graph(graph, stream=s):
            g.run(stream=s)
    for _ in range(2):
        graph.replay()
        torch.cuda.synchronize()
        gk, gv = g.gather()
        np.testing.assert_array_equal(gk, ek)
        np.testing.assert_array_equal(gv, ev)
    assert g.status() == 0


def test_two_translators_on_two_streams():
    """Two translations in flight at once on two streams write exactly their eager results."""
    a = make_case(_shrink(SPECS["qwen7b_to_qwen1p5b_4k"], 2, 2), [640])
    b = make_case(_shrink(SPECS["llama70b_to_qwen7b_8k"], 5, 3), [500])
    ga, gb = _run(a, kvx.KVX_PATH_AUTO), _run(b, kvx.KVX_PATH_AUTO)
    ref = (ga.gather(), gb.gather())
    for g in (ga, gb):
        for t in g.dst_k + g.dst_v:
            t.fill_(float("nan"))
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    s1.wait_stream(torch.cuda.current_stream())
    s2.wait_stream(torch.cuda.current_stream())
    for _ in range(3):
        ga.run(stream=s1)
        gb.run(stream=s2)
    torch.cuda.synchronize()
    for g, (rk, rv) in zip((ga, gb), ref):
        gk, gv = g.gather()
        np.testing.assert_array_equal(gk, rk)
        np.testing.assert_array_equal(gv, rv)
        assert g.status() == 0


# ------------------------------------------------------------------ limits of the fast paths
@pytest.mark.parametrize("batch", [300, 600])
def test_large_batches(batch):
    """More sequences than the identity kernel keeps on chip (256), and than the span kernel
    caches in shared memory (512): both fall back to their general paths, same results."""
    rng = np.random.default_rng(batch)
    lens = [int(x) for x in rng.integers(1, 24, size=batch)]
    for base in ("qwen7b_to_qwen1p5b_4k", "qwen1p5b_to_gemma2b_1k"):
        spec = _shrink(SPECS[base], 2, 2)
        c = make_case(spec, lens)
        g, _, _ = _full_compare(c, kvx.KVX_PATH_AUTO)
        assert g.tr.info().path == kvx.KVX_PATH_TCGEN05


def test_more_target_layers_than_the_identity_kernel_takes():
    """100 target layers (above the identity kernel's 96): the span kernel serves identity
    alignment too."""
    spec = synth.WorkloadSpec("deep", synth.ModelGeom(120, 2, 64, 1e4), synth.ModelGeom(100, 1, 64, 1e6), "bf16",
                              [40], False, None, False)
    c = make_case(spec, [40, 17])
    _full_compare(c, kvx.KVX_PATH_AUTO)
