"""The closed-form translator fit (kvx_fit_*) against the oracle's fit, through the C ABI.

W is compared element by element against a bound derived from the two sides' arithmetic
(_elementwise_bound), and also through rel-L2 and recovery of a planted translator.

The oracle solves the normal equations in double from exact span means; the library rounds
the input rows X and the target rows Y to the cache dtype and sums X^T X, X^T Y in fp32.
Tolerance for bf16: the rounding of X and Y is about 2^-9 / sqrt(3) ~ 1.1e-3 relative (RMS),
and least squares amplifies it by cond(X) ~ (1 + sqrt(in/T)) / (1 - sqrt(in/T)), 2.4 at
in = 256, T = 1500: ~3e-3 relative on W, so rel-L2 <= 1e-2.  fp32 caches: 1e-4.
"""
import dataclasses

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle
import paper_2608_30963_gb300 as kvx
from paper_2608_30963_gb300 import synth

from harness import make_case, oracle_problem

pytestmark = pytest.mark.gpu
SPECS = synth.config_specs()


@pytest.fixture(scope="module", autouse=True)
def _lib():
    kvx.build()
    yield


def _shrink(spec, Ls, Lt, **kw):
    return dataclasses.replace(spec, src=dataclasses.replace(spec.src, num_layers=Ls),
                               dst=dataclasses.replace(spec.dst, num_layers=Lt), **kw)


def _rel(a, b):
    return float(np.linalg.norm(np.asarray(a, np.float64) - b) / np.linalg.norm(b))


def _targets_from(c, wk, wv):
    """The target model's 'own' caches: the oracle's translation with planted weights,
    stored in the cache dtype, per target layer [B, Ht, t_max, dt]."""
    p = oracle_problem(dataclasses.replace(c, w_k=wk, w_v=wv))
    ok, ov = p.translate()                                   # [Lt, Ht, T, dt]
    wl, s = c.wl, c.spec
    Lt, Ht, dt = s.dst.num_layers, s.dst.num_kv_heads, s.dst.head_dim
    tk = np.zeros((Lt, wl.batch, Ht, max(wl.t_max, 1), dt), np.float32)
    tv = np.zeros_like(tk)
    for b in range(wl.batch):
        a, e = int(wl.tgt_seq_off[b]), int(wl.tgt_seq_off[b + 1])
        tk[:, b, :, :e - a] = ok[:, :, a:e]
        tv[:, b, :, :e - a] = ov[:, :, a:e]
    if s.dtype == "bf16":
        tk, tv = synth.bf16_round(tk), synth.bf16_round(tv)
    return tk, tv


def _elementwise_bound(c, tk, tv, lam, wk_ref, wv_ref, chol_u=2.0 ** -24):
    """Per-element bound on |W_gpu - W_oracle| from the arithmetic of the two sides.

    The oracle solves (X^T X + lam I) W = X^T Y in double from exact input rows X.  The library
    rounds X (and, for K, the un-rotated target rows Y) to the cache dtype, sums X^T X and X^T Y
    over the T tokens in fp32 and factors in fp32 (or double).  To first order, with A = (X^T X + lam I)^-1,
    P = A X^T and the residual R = Y - X W:
        dW = A dX^T R - P dX W + P dY  (+ the effect of the fp32 sums and factorisation).
    Rounding to nearest leaves independent errors |dX_tk| <= u |X_tk| of variance u^2 X_tk^2 / 3
    (u = 2^-8 for bf16), so each element of dW has the standard deviation
        sigma = sqrt(u^2/3 [A^2 (X^2)^T R^2]) + sqrt(u^2/3 [P^2 X^2 W^2]) (+) sqrt(u_y^2/3 [P^2 Y^2])
    (squares elementwise, products matrix products; the first two share dX and are added, the
    third in quadrature).  The fp32 sums of T terms add, with the probabilistic rounding-error
    bound of Higham and Mary (confidence factor 6), at most gamma = 6 sqrt(T) 2^-24 relative to
    the sums of |terms|, and the Cholesky factorisation a backward error of about 3 in u_c |G|
    (u_c = 2^-24 for the fp32 factor, 2^-53 where the library factors in double):
        gamma |A| (|X|^T |Y| + |X|^T |X| |W|) + 3 in u_c |A| |G| |W|.
    The bound is 6 sigma plus those terms, per (layer, head, K|V) group."""
    s = c.spec
    p = oracle_problem(c)
    wl = c.wl
    T = wl.total_tgt
    bf = s.dtype == "bf16"
    u = 2.0 ** -8 if bf else 4 * 2.0 ** -24
    gamma = 6 * np.sqrt(T) * 2.0 ** -24
    din, dt = s.group_in, s.dst.head_dim
    seq = np.searchsorted(wl.tgt_seq_off, np.arange(T), side="right") - 1
    out = []
    for kv, tgt, wref in ((0, tk, wk_ref), (1, tv, wv_ref)):
        bk = np.zeros_like(wref)
        for j in range(s.dst.num_layers):
            for h in range(s.dst.num_kv_heads):
                X = np.stack([p.input_row(j, h, kv, tp) for tp in range(T)])
                Y = np.empty((T, dt))
                for tp in range(T):
                    b = int(seq[tp])
                    t = tp - int(wl.tgt_seq_off[b])
                    y = np.asarray(tgt[j][b, h, t], np.float64)
                    pt = float(t if c.tgt_pos is None else c.tgt_pos[tp])
                    Y[tp] = oracle.rope_g(y, s.dst, pt, -1) if kv == 0 and s.dst.rope_base > 0 else y
                W = wref[j, h]
                G = X.T @ X + lam * np.eye(din)
                A = np.linalg.inv(G)
                P = A @ X.T
                R = Y - X @ W
                u_y = u if (kv == 0 or not bf) else 0.0
                s1 = np.sqrt(u * u / 3 * ((A * A) @ ((X * X).T @ (R * R))))
                s3 = np.sqrt(u * u / 3 * ((P * P) @ ((X * X) @ (W * W))))
                s2 = np.sqrt(u_y * u_y / 3 * ((P * P) @ (Y * Y)))
                sigma = np.sqrt((s1 + s3) ** 2 + s2 ** 2)
                aX, aW, aA = np.abs(X), np.abs(W), np.abs(A)
                bk[j, h] = (6 * sigma + gamma * (aA @ (aX.T @ np.abs(Y) + (aX.T @ aX) @ aW))
                            + 3 * din * chol_u * (aA @ (np.abs(G) @ aW)))
        out.append(bk)
    return out


def _assert_elementwise(gpu, ref, bound, label):
    err = np.abs(np.asarray(gpu, np.float64) - ref)
    bad = err > bound
    worst = float((err / np.maximum(bound, 1e-300)).max())
    print(f"fit {label}: max |dW| {err.max():.3e}, worst |dW| / bound {worst:.3f}, max bound {bound.max():.3e}")
    assert not bad.any(), (label, int(bad.sum()), worst)


def _fit_gpu(c, tk, tv, lam, chunk=0, split=None, paged=False):
    from gpu_harness import DeviceCase, to_dev, i32
    s = c.spec
    g = DeviceCase(c, path=kvx.KVX_PATH_SIMT, paged=False)     # device source buffers and metadata
    dtk = [to_dev(tk[j], s.dtype) for j in range(s.dst.num_layers)]
    dtv = [to_dev(tv[j], s.dtype) for j in range(s.dst.num_layers)]
    f = kvx.Fitter(s.src, s.dst, lam, layer_map=c.layer_map.tolist(), dtype=g.tr.desc.dtype, form=s.form,
                   layers_per_target=s.layers_per_target, chunk_tokens=chunk)
    wl = c.wl
    kw = dict(span_lo=g.span_lo, span_hi=g.span_hi, src_pos=g.src_pos, tgt_pos=g.tgt_pos)
    if paged:
        P = s.page_size
        pages = [(int(t) + P - 1) // P for t in wl.tgt_len]
        npg, mp = sum(pages), max(pages)
        perm = np.random.default_rng(9).permutation(npg).astype(np.int32)
        pt = np.full((wl.batch, mp), -1, np.int32)
        k = 0
        for b, n in enumerate(pages):
            pt[b, :n] = perm[k:k + n]; k += n
        pool_k = [torch.zeros((npg, P, s.dst.num_kv_heads, s.dst.head_dim), dtype=dtk[0].dtype, device="cuda")
                  for _ in dtk]
        pool_v = [torch.zeros_like(x) for x in pool_k]
        for j in range(s.dst.num_layers):
            for b in range(wl.batch):
                for t in range(int(wl.tgt_len[b])):
                    pool_k[j][pt[b, t // P], t % P] = dtk[j][b, :, t]
                    pool_v[j][pt[b, t // P], t % P] = dtv[j][b, :, t]
        dtk, dtv = pool_k, pool_v
        kw.update(page_table=i32(pt), page_size=P, num_pages=npg)
    if split is None:
        f.accumulate(g.src_k, g.src_v, g.src_len, g.seq_off, wl.total_tgt, dtk, dtv, **kw)
    else:
        # two calibration calls over sequences [0, split) and [split, B)
        for lo, hi in ((0, split), (split, wl.batch)):
            a, e = int(wl.tgt_seq_off[lo]), int(wl.tgt_seq_off[hi])
            sk = [x[lo:hi] for x in g.src_k]
            sv = [x[lo:hi] for x in g.src_v]
            off = i32(wl.tgt_seq_off[lo:hi + 1] - a)
            kws = dict(span_lo=None if g.span_lo is None else g.span_lo[a:e],
                       span_hi=None if g.span_hi is None else g.span_hi[a:e])
            f.accumulate(sk, sv, g.src_len[lo:hi], off, e - a, [x[lo:hi] for x in dtk], [x[lo:hi] for x in dtv],
                         **kws)
    in_dim = s.group_in
    tdt = torch.bfloat16 if s.dtype == "bf16" else torch.float32
    wk = torch.empty((s.dst.num_layers, s.dst.num_kv_heads, in_dim, s.dst.head_dim), dtype=tdt, device="cuda")
    wv = torch.empty_like(wk)
    bits = f.solve(wk, wv)
    assert f.tokens() == wl.total_tgt
    from gpu_harness import to_host
    return to_host(wk), to_host(wv), bits, f


CASES = {
    # name: (base spec, Ls, Lt, target lengths, extra spec fields)
    "qwen7b_qwen1p5b_identity": ("qwen7b_to_qwen1p5b_4k", 3, 2, [900, 600], {}),
    "gemma_expansion_spans": ("qwen1p5b_to_gemma2b_1k", 3, 2, [700, 500], {}),
    # partial rotary heads on both sides (a half of the source head, a quarter of the target's)
    "partial_rotary_identity": ("qwen7b_to_qwen1p5b_4k", 3, 2, [900, 600],
                                dict(src=synth.ModelGeom(3, 4, 128, 1e6, rotary_dim=64),
                                     dst=synth.ModelGeom(2, 2, 128, 1e6, rotary_dim=32))),
    # dense per-layer form over 2 source heads of 128 (in = 256), cross-tokenizer spans
    # 64-channel heads: in = 64 is not a multiple of the tensor-core row block (128), so the
    # CUDA-core Gram path runs on bf16 caches
    "small_heads_cuda_core": ("qwen7b_to_qwen1p5b_4k", 3, 2, [900, 300], dict(src=synth.ModelGeom(3, 2, 64, 1e6),
                                                                             dst=synth.ModelGeom(2, 2, 64, 1e4))),
    "dense_spans": ("llama70b_to_qwen7b_8k", 4, 2, [1100, 700], dict(form=synth.FORM_DENSE,
                                                                   src=synth.ModelGeom(4, 2, 128, 5e5),
                                                                   dst=synth.ModelGeom(2, 2, 64, 1e6))),
}


@pytest.mark.parametrize("name", list(CASES))
def test_fit_recovers_planted_translator_and_matches_oracle(name):
    base, Ls, Lt, lens, kw = CASES[name]
    spec = _shrink(SPECS[base], Ls, Lt)
    if "dst" in kw:
        kw = dict(kw, dst=dataclasses.replace(kw["dst"], num_layers=Lt))
    if "src" in kw:
        kw = dict(kw, src=dataclasses.replace(kw["src"], num_layers=Ls))
    spec = dataclasses.replace(spec, **kw)
    c = make_case(spec, lens)
    rng = np.random.default_rng(17)
    din, dt = spec.group_in, spec.dst.head_dim
    w_true = [synth.bf16_round(rng.standard_normal((Lt, spec.dst.num_kv_heads, din, dt)).astype(np.float32)
                               / np.float32(np.sqrt(din))) for _ in range(2)]
    tk, tv = _targets_from(c, *w_true)
    lam = 1e-3
    gk, gv, bits, _ = _fit_gpu(c, tk, tv, lam)
    assert bits == 0
    ok, ov = oracle_problem(c).fit(list(tk), list(tv), lam)
    bk, bv = _elementwise_bound(c, tk, tv, lam, ok, ov)
    for gpu, ref, true, bound, lab in ((gk, ok, w_true[0], bk, "K"), (gv, ov, w_true[1], bv, "V")):
        assert np.all(np.isfinite(gpu))
        _assert_elementwise(gpu, ref, bound, f"{name} {lab}")
        assert _rel(gpu, ref) <= 1e-2, _rel(gpu, ref)
        assert _rel(gpu, true) <= 1e-2, _rel(gpu, true)
        assert _rel(ref, true) <= 5e-3, _rel(ref, true)


def test_fit_with_explicit_positions_matches_oracle():
    """Identity alignment with position arrays on both sides: source rows at s + 3b, target rows
    at t + 3b for even t and t + 3b + 7 for odd t, so half the tokens share their source
    rotation with the target's and half do not.  Both rotations are the same schedule here
    (7B -> 1.5B shapes), the case where one (cos, sin) may serve both sides of a token."""
    spec = _shrink(SPECS["qwen7b_to_qwen1p5b_4k"], 3, 2)
    lens = [700, 500]
    wl = synth.make_workload(spec, lens)
    src_pos = np.stack([np.arange(wl.s_max) + 3 * b for b in range(wl.batch)]).astype(np.int32)
    tgt_pos = np.empty(wl.total_tgt, np.int32)
    for b in range(wl.batch):
        a, e = int(wl.tgt_seq_off[b]), int(wl.tgt_seq_off[b + 1])
        t = np.arange(e - a)
        tgt_pos[a:e] = t + 3 * b + 7 * (t & 1)
    c = make_case(spec, lens, src_pos=src_pos, tgt_pos=tgt_pos, wl=wl)
    rng = np.random.default_rng(23)
    din, dt = spec.group_in, spec.dst.head_dim
    w_true = [synth.bf16_round(rng.standard_normal((2, spec.dst.num_kv_heads, din, dt)).astype(np.float32)
                               / np.float32(np.sqrt(din))) for _ in range(2)]
    tk, tv = _targets_from(c, *w_true)
    lam = 1e-3
    gk, gv, bits, _ = _fit_gpu(c, tk, tv, lam)
    assert bits == 0
    ok, ov = oracle_problem(c).fit(list(tk), list(tv), lam)
    bk, bv = _elementwise_bound(c, tk, tv, lam, ok, ov)
    for gpu, ref, true, bound, lab in ((gk, ok, w_true[0], bk, "K"), (gv, ov, w_true[1], bv, "V")):
        _assert_elementwise(gpu, ref, bound, f"positions {lab}")
        assert _rel(gpu, true) <= 1e-2, _rel(gpu, true)


def test_fit_fp32_tiny_matches_oracle_tightly():
    spec = SPECS["tiny_fp32"]
    c = make_case(spec, [256, 200])
    rng = np.random.default_rng(18)
    tk = rng.standard_normal((2, 2, 1, 256, 64)).astype(np.float32)   # unrelated targets: a genuine fit
    tv = rng.standard_normal((2, 2, 1, 256, 64)).astype(np.float32)
    lam = 0.5
    gk, gv, bits, _ = _fit_gpu(c, tk, tv, lam)
    ok, ov = oracle_problem(c).fit(list(tk), list(tv), lam)
    assert bits == 0
    bk, bv = _elementwise_bound(c, tk, tv, lam, ok, ov)
    _assert_elementwise(gk, ok, bk, "tiny fp32 K")
    _assert_elementwise(gv, ov, bv, "tiny fp32 V")
    assert _rel(gk, ok) <= 1e-4 and _rel(gv, ov) <= 1e-4


def test_fit_ill_conditioned_calibration_matches_oracle():
    """A calibration set whose two source heads nearly coincide (head 1 = head 0 + 3e-3 noise):
    X^T X + lambda I has a condition number above 1e6, where an fp32 Cholesky factor loses most
    of its digits.  The fitter sees it in the factor's pivots and factors those systems again in
    double (status bit 0x40); W then matches the oracle's fp64 solution within the bound of the
    fp32 sums and a double factorisation.  fp32 caches, so the rows carry no bf16 rounding."""
    spec = SPECS["tiny_fp32"]
    c = make_case(spec, [456])
    rng = np.random.default_rng(21)
    for d in (c.src_k, c.src_v):
        for l in d:
            d[l][:, 1] = d[l][:, 0] + np.float32(3e-3) * rng.standard_normal(d[l][:, 0].shape).astype(np.float32)
    w_true = [rng.standard_normal((2, 1, 128, 64)).astype(np.float32) / np.float32(np.sqrt(128)) for _ in range(2)]
    tk, tv = _targets_from(c, *w_true)
    tk = tk + np.float32(1e-3) * rng.standard_normal(tk.shape).astype(np.float32)   # not an exact fit
    tv = tv + np.float32(1e-3) * rng.standard_normal(tv.shape).astype(np.float32)
    lam = 1e-4
    gk, gv, bits, _ = _fit_gpu(c, tk, tv, lam)
    assert bits & 0x40, f"status 0x{bits:x}: no system was solved in double"
    assert not bits & 0x20
    ok, ov = oracle_problem(c).fit(list(tk), list(tv), lam)
    p = oracle_problem(c)
    X = np.stack([p.input_row(0, 0, 0, tp) for tp in range(c.wl.total_tgt)])
    ev = np.linalg.eigvalsh(X.T @ X + lam * np.eye(X.shape[1]))
    print(f"ill-conditioned fit: cond(X^T X + lambda I) = {ev[-1] / ev[0]:.3e}")
    assert ev[-1] / ev[0] > 1e6
    bk, bv = _elementwise_bound(c, tk, tv, lam, ok, ov, chol_u=2.0 ** -53)
    _assert_elementwise(gk, ok, bk, "ill-conditioned K")
    _assert_elementwise(gv, ov, bv, "ill-conditioned V")


def test_fit_two_calls_chunked_and_paged_agree_with_one_call():
    """Sums over calibration calls and accumulation passes add up: one call, two calls, a
    small chunk (several passes) and a paged target cache give the same W (fp32 summation
    order only)."""
    spec = _shrink(SPECS["qwen1p5b_to_gemma2b_1k"], 2, 2)
    c = make_case(spec, [500, 300, 400])
    rng = np.random.default_rng(19)
    w_true = [synth.bf16_round(rng.standard_normal((2, 4, 128, 256)).astype(np.float32) / np.float32(np.sqrt(128)))
              for _ in range(2)]
    tk, tv = _targets_from(c, *w_true)
    one_k, one_v, _, f = _fit_gpu(c, tk, tv, 1e-2)
    for kw in (dict(split=1), dict(chunk=160), dict(paged=True)):
        k2, v2, bits, _ = _fit_gpu(c, tk, tv, 1e-2, **kw)
        assert bits == 0
        assert _rel(k2, one_k) <= 2e-3 and _rel(v2, one_v) <= 2e-3, kw
    # reset: a second fit from the same fitter after reset equals the first
    f.reset()
    assert f.tokens() == 0


def test_fitted_translator_reproduces_the_targets():
    """End to end: fit on a calibration context, build a translator from the fitted W and
    translate the same context: the output is the target cache up to bf16 rounding."""
    from gpu_harness import DeviceCase, to_dev
    from harness import compare
    spec = _shrink(SPECS["qwen7b_to_qwen1p5b_4k"], 2, 2)
    c = make_case(spec, [1200])
    rng = np.random.default_rng(20)
    w_true = [synth.bf16_round(rng.standard_normal((2, 2, 256, 128)).astype(np.float32) / np.float32(16.0))
              for _ in range(2)]
    tk, tv = _targets_from(c, *w_true)
    gk, gv, bits, _ = _fit_gpu(c, tk, tv, 1e-3)
    fitted = dataclasses.replace(c, w_k=synth.bf16_round(gk), w_v=synth.bf16_round(gv))
    g = DeviceCase(fitted)
    g.run()
    torch.cuda.synchronize()
    outk, outv = g.gather()
    ref_k = np.stack([tk[j][0] for j in range(2)])    # [Lt, Ht, T, dt]
    ref_v = np.stack([tv[j][0] for j in range(2)])
    compare(outk, ref_k, "bf16")
    compare(outv, ref_v, "bf16")
