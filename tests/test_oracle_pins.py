"""Pins for the CPU oracle, independent of its own code.

Each test checks the oracle against something the mathematics fixes: brute
force on tiny inputs, closed forms, invariants, or special cases that reduce to
a library routine.  Between them a dropped term, a wrong sign, a wrong index or
a transposed operand anywhere in the oracle fails at least one test.
"""
from fractions import Fraction

import numpy as np
import pytest

import oracle
from paper_2608_30963_gb300 import synth


# ---------------------------------------------------------------- layer map
@pytest.mark.parametrize("Ls,Lt", [(4, 2), (28, 28), (28, 26), (80, 28), (5, 3), (3, 5), (7, 1), (1, 4), (2, 2),
                                   (10, 4)])
def test_layer_map_matches_exact_nearest_depth(Ls, Lt):
    got = oracle.layer_map_nearest(Ls, Lt)
    for j in range(Lt):
        dj = Fraction(j, Lt - 1) if Lt > 1 else Fraction(0)
        cands = [abs(Fraction(s, Ls - 1) - dj) if Ls > 1 else Fraction(0) for s in range(Ls)]
        m = min(cands)
        best = max(s for s in range(Ls) if cands[s] == m)  # ties go to the deeper layer
        assert got[j] == best


def test_layer_map_endpoints_and_identity():
    assert list(oracle.layer_map_nearest(28, 28)) == list(range(28))
    for Ls, Lt in [(80, 28), (28, 26), (4, 2)]:
        m = oracle.layer_map_nearest(Ls, Lt)
        assert m[0] == 0 and m[-1] == Ls - 1
        assert np.all(np.diff(m) > 0)


# ---------------------------------------------------------- token alignment
def test_alignment_recovers_generated_partition():
    for b, T in enumerate([1, 7, 300, 2048]):
        lo, hi, S, se, te = synth.draw_spans(T, b)
        so = np.array([0, S], np.int32)
        to = np.array([0, T], np.int32)
        glo, ghi, n = oracle.build_alignment(so, se, to, te)
        assert n == 0
        np.testing.assert_array_equal(glo, lo)
        np.testing.assert_array_equal(ghi, hi)


def _bytewise_spans(src_end, tgt_end):
    """Brute force over bytes: owner of each byte in both tokenisations."""
    n = int(src_end[-1])
    src_of = np.searchsorted(src_end, np.arange(n), side="right")
    tgt_of = np.searchsorted(tgt_end, np.arange(n), side="right")
    members = [[] for _ in range(len(tgt_end))]
    for s in range(len(src_end)):
        members[tgt_of[int(src_end[s]) - 1]].append(s)   # s's last byte
    lo, hi = [], []
    for t in range(len(tgt_end)):
        if members[t]:
            assert members[t] == list(range(members[t][0], members[t][-1] + 1))
            lo.append(members[t][0]); hi.append(members[t][-1] + 1)
        else:
            s = int(src_of[int(tgt_end[t]) - 1])            # holds t's last byte
            lo.append(s); hi.append(s + 1)
    return np.array(lo, np.int32), np.array(hi, np.int32)


@pytest.mark.parametrize("key,ms,mt", [(0, 4.0, 4.0), (1, 5.0, 2.0), (2, 2.0, 6.0), (3, 1.0, 3.0), (4, 3.0, 1.0)])
def test_alignment_bytewise_bruteforce(key, ms, mt):
    # batch of 3 sequences of different byte lengths, including empty spans
    src_ends, tgt_ends = [], []
    for i, nb in enumerate([1, 57, 911]):
        se, te = synth.draw_tokenizations(nb, ms, mt, key * 10 + i)
        src_ends.append(se); tgt_ends.append(te)
    so = np.concatenate([[0], np.cumsum([len(x) for x in src_ends])]).astype(np.int32)
    to = np.concatenate([[0], np.cumsum([len(x) for x in tgt_ends])]).astype(np.int32)
    lo, hi, n = oracle.build_alignment(so, np.concatenate(src_ends), to, np.concatenate(tgt_ends))
    assert n == 0
    for b in range(3):
        elo, ehi = _bytewise_spans(src_ends[b], tgt_ends[b])
        np.testing.assert_array_equal(lo[to[b]:to[b + 1]], elo)
        np.testing.assert_array_equal(hi[to[b]:to[b + 1]], ehi)


# --------------------------------------------------------------------- RoPE
def test_rope_two_dims_is_plain_rotation_by_position():
    # d = 2: the only frequency is base^0 = 1, so the angle is the position.
    for base in (10.0, 1e4, 1e6):
        y = oracle.rope(np.array([1.0, 0.0]), base, np.pi / 2, +1)
        np.testing.assert_allclose(y, [0.0, 1.0], atol=1e-15)
        y = oracle.rope(np.array([0.0, 2.0]), base, np.pi, +1)
        np.testing.assert_allclose(y, [0.0, -2.0], atol=1e-14)


def test_rope_roformer_frequencies_d4():
    # RoFormer: theta_i = base^(-2(i-1)/d), i = 1..d/2; d = 4, base 1e4 -> {1, 1e-2}.
    x = np.array([0.0, 1.0, 0.0, 0.0])     # unit vector in the second (slow) pair
    y = oracle.rope(x, 1e4, 100.0, +1)     # angle 100 * 1e-2 = 1 rad
    np.testing.assert_allclose(y, [0.0, np.cos(1.0), 0.0, np.sin(1.0)], atol=1e-14)


def test_rope_equals_complex_multiplication():
    rng = np.random.default_rng(11)
    for d in (2, 8, 64, 128, 256):
        for base, pos in ((1e4, 3.0), (1e6, 4095.0), (5e5, 31999.0)):
            x = rng.standard_normal(d)
            h = d // 2
            z = x[:h] + 1j * x[h:]
            ang = pos * np.exp(-np.log(base) * np.arange(0, d, 2) / d)
            w = z * np.exp(1j * ang)
            y = oracle.rope(x, base, pos, +1)
            np.testing.assert_allclose(y, np.concatenate([w.real, w.imag]), rtol=0, atol=1e-9)


def _complex_rope(x, base, pos, d_rot=None, scale=1.0):
    """Half-split RoPE by complex multiplication: pairs (i, i + n/2) of the first n channels as
    z_i = x_i + 1j x_{i+n/2}, turned by (pos / scale) * base^(-2i/n); other channels unchanged."""
    d = x.shape[-1]
    n = d if d_rot is None else d_rot
    h = n // 2
    z = x[..., :h].astype(np.float64) + 1j * x[..., h:n].astype(np.float64)
    ang = (np.asarray(pos, np.float64)[..., None] / scale) * np.power(float(base), -2.0 * np.arange(h) / n)
    w = z * np.exp(1j * ang)
    return np.concatenate([w.real, w.imag, x[..., n:].astype(np.float64)], axis=-1)


def test_rope_cache_rotates_each_row_at_its_own_position():
    """The input-synthesis rotation of whole caches: row (b, h, s) turns by the position of
    token s of sequence b, 0..S-1 without a position array, pos[b, s] with one, backwards for
    sign -1; and under a schedule it equals the single-row map at the same position."""
    rng = np.random.default_rng(13)
    B, H, S, d = 2, 3, 40, 64
    x = rng.standard_normal((B, H, S, d)).astype(np.float32)
    base = 1e4
    pos = rng.permutation(np.arange(5, 5 + B * S)).reshape(B, S).astype(np.int32) * 37
    # default positions: token index
    y = oracle.rope_cache(x, base)
    np.testing.assert_allclose(y, _complex_rope(x, base, np.arange(S)[None, None, :]), rtol=0, atol=2e-6)
    # explicit positions, per sequence and token, shared by the heads
    yp = oracle.rope_cache(x, base, pos)
    np.testing.assert_allclose(yp, _complex_rope(x, base, pos[:, None, :]), rtol=0, atol=2e-6)
    assert np.abs(yp - y).max() > 0.1        # the position array is used
    # sign -1 turns backwards, so it undoes sign +1 at the same positions
    ym = oracle.rope_cache(x, base, pos, -1)
    np.testing.assert_allclose(ym, _complex_rope(x, base, -pos[:, None, :]), rtol=0, atol=2e-6)
    # schedules and partial rotary heads: row by row the single-row map (itself pinned above)
    geoms = [synth.ModelGeom(1, H, d, 1e4, rope_type=synth.ROPE_LINEAR, rope_factor=4.0),
             synth.ModelGeom(1, H, d, 1e4, rotary_dim=32), synth.LLAMA70B_SCALED]
    for g in geoms:
        xg = x if g.head_dim == d else rng.standard_normal((B, H, S, g.head_dim)).astype(np.float32)
        yg = oracle.rope_cache(xg, g, pos)
        for b in range(B):
            for hh in range(H):
                for s_ in (0, 1, S // 2, S - 1):
                    ref = oracle.rope_g(xg[b, hh, s_], g, float(pos[b, s_]), +1)
                    np.testing.assert_allclose(yg[b, hh, s_], ref, rtol=0, atol=4e-6)
    # the linear schedule is plain RoPE at pos / factor; the partial head rotates its first 32 channels
    lin = oracle.rope_cache(x, geoms[0], pos)
    np.testing.assert_allclose(lin, _complex_rope(x, 1e4, pos[:, None, :], scale=4.0), rtol=0, atol=2e-6)
    part = oracle.rope_cache(x, geoms[1], pos)
    np.testing.assert_allclose(part, _complex_rope(x, 1e4, pos[:, None, :], d_rot=32), rtol=0, atol=2e-6)


def test_rope_inverse_norm_and_relative_position():
    rng = np.random.default_rng(12)
    for d, base in ((64, 1e4), (128, 1e6), (256, 1e4)):
        x = rng.standard_normal(d)
        q = rng.standard_normal(d)
        back = oracle.rope(oracle.rope(x, base, 777.0, +1), base, 777.0, -1)
        np.testing.assert_allclose(back, x, atol=1e-12)
        np.testing.assert_array_equal(oracle.rope(x, base, 0.0, +1), x)
        y = oracle.rope(x, base, 1234.0, +1)
        h = d // 2
        np.testing.assert_allclose(x[:h] ** 2 + x[h:] ** 2, y[:h] ** 2 + y[h:] ** 2, rtol=1e-12)
        # <R(p)q, R(p')k> depends only on p - p'
        a = oracle.rope(q, base, 100.0, +1) @ oracle.rope(x, base, 40.0, +1)
        b = oracle.rope(q, base, 1160.0, +1) @ oracle.rope(x, base, 1100.0, +1)
        assert abs(a - b) < 1e-9


# ------------------------------------------------- RoPE frequency schedules
def _sched(base, d=4, **kw):
    return synth.ModelGeom(1, 1, d, base, **kw)


def _slow_pair_angle(g, pos=1.0):
    """Angle by which the second pair of a d=4 head turns at `pos` (theta_1 = base^(-1/2))."""
    y = oracle.rope_g(np.array([0.0, 1.0, 0.0, 0.0]), g, pos, +1)
    return np.arctan2(y[3], y[1])


def test_linear_schedule_is_position_interpolation():
    # angle of position p under factor F equals the plain angle of position p / F
    rng = np.random.default_rng(21)
    for d, base, F in ((64, 1e4, 2.0), (128, 1e6, 4.0), (256, 1e4, 8.0)):
        x = rng.standard_normal(d)
        g = synth.ModelGeom(1, 1, d, base, rope_type=synth.ROPE_LINEAR, rope_factor=F)
        for p in (1.0, 37.0, 4095.0):
            np.testing.assert_allclose(oracle.rope_g(x, g, p, +1), oracle.rope(x, base, p / F, +1), atol=1e-9)


def test_llama3_schedule_factor_one_is_plain():
    rng = np.random.default_rng(22)
    x = rng.standard_normal(128)
    g = synth.ModelGeom(1, 1, 128, 5e5, rope_type=synth.ROPE_LLAMA3, rope_factor=1.0,
                        rope_low_freq_factor=1.0, rope_high_freq_factor=4.0, rope_original_max_position=8192)
    np.testing.assert_allclose(oracle.rope_g(x, g, 3000.0, +1), oracle.rope(x, 5e5, 3000.0, +1), atol=1e-12)


def test_llama3_schedule_bands_and_continuity():
    # d = 4: the slow pair's wavelength is 2 pi sqrt(base), so base places it anywhere.
    F, lo, hi, orig = 8.0, 1.0, 4.0, 8192
    kw = dict(rope_type=synth.ROPE_LLAMA3, rope_factor=F, rope_low_freq_factor=lo,
              rope_high_freq_factor=hi, rope_original_max_position=orig)
    base_of = lambda w: (w / (2 * np.pi)) ** 2
    theta = lambda w: 2 * np.pi / w
    short_edge, long_edge = orig / hi, orig / lo           # 2048 and 8192 tokens
    # short wavelengths keep their frequency, long ones are divided by the factor
    for w in (100.0, 2000.0):
        assert _slow_pair_angle(_sched(base_of(w), **kw)) == pytest.approx(theta(w), rel=1e-12)
    for w in (8300.0, 1e6):
        assert _slow_pair_angle(_sched(base_of(w), **kw)) == pytest.approx(theta(w) / F, rel=1e-12)
    # continuous at both band edges
    for edge, inside in ((short_edge, theta(short_edge)), (long_edge, theta(long_edge) / F)):
        a = _slow_pair_angle(_sched(base_of(edge * (1 - 1e-9)), **kw))
        b = _slow_pair_angle(_sched(base_of(edge * (1 + 1e-9)), **kw))
        assert a == pytest.approx(inside, rel=1e-6) and b == pytest.approx(inside, rel=1e-6)
    # inside the band the frequency lies strictly between theta/F and theta and falls with w
    ws = np.linspace(short_edge * 1.01, long_edge * 0.99, 9)
    ang = np.array([_slow_pair_angle(_sched(base_of(w), **kw)) for w in ws])
    assert np.all(ang < theta(ws)) and np.all(ang > theta(ws) / F) and np.all(np.diff(ang) < 0)
    # where orig / w sits halfway between low and high the two frequencies weigh equally
    w_mid = orig / ((lo + hi) / 2)
    assert _slow_pair_angle(_sched(base_of(w_mid), **kw)) == pytest.approx(theta(w_mid) * (1 + 1 / F) / 2,
                                                                            rel=1e-12)
    # the fast pair (theta_0 = 1, wavelength 2 pi) is never rescaled
    y = oracle.rope_g(np.array([1.0, 0.0, 0.0, 0.0]), _sched(1e9, **kw), 0.5, +1)
    assert np.arctan2(y[2], y[0]) == pytest.approx(0.5, rel=1e-14)


def test_llama31_parameters_split_128_dim_heads_29_6_29():
    # base 5e5, d 128: wavelength 2 pi 5e5^(i/64) is below 2048 for i <= 28 and above 8192
    # for i >= 35 (ln(2048/2pi)/ln(5e5)*64 = 28.2, ln(8192/2pi)/ln(5e5)*64 = 35.0)
    g = synth.LLAMA70B_SCALED
    kept = scaled = mixed = 0
    for i in range(64):
        x = np.zeros(128)
        x[i] = 1.0
        p = 0.25                                   # keeps every angle below pi
        y = oracle.rope_g(x, g, p, +1)
        got = np.arctan2(y[i + 64], y[i]) / p
        plain = 5e5 ** (-i / 64)
        if got == pytest.approx(plain, rel=1e-12):
            kept += 1
        elif got == pytest.approx(plain / 8, rel=1e-12):
            scaled += 1
        else:
            assert plain / 8 < got < plain
            mixed += 1
    assert (kept, mixed, scaled) == (29, 6, 29)


def test_scheduled_translation_undoes_and_reapplies_the_schedule():
    # K stored with a scheduled source RoPE, W = I, identity alignment and the same scheduled
    # target RoPE: the translation returns the stored keys (un-rotate then re-rotate).
    g = synth.ModelGeom(1, 1, 64, 5e5, rope_type=synth.ROPE_LLAMA3, rope_factor=8.0,
                        rope_low_freq_factor=1.0, rope_high_freq_factor=4.0, rope_original_max_position=64)
    rng = np.random.default_rng(23)
    S = 40
    k = oracle.rope_cache(rng.standard_normal((1, 1, S, 64)).astype(np.float32), g)
    v = rng.standard_normal((1, 1, S, 64)).astype(np.float32)
    W = np.eye(64, dtype=np.float32)[None, None]
    p = oracle.OracleProblem(g, g, [0], [S], [0, S], S, S, [k], [v], W, W)
    ok, ov = p.translate()
    np.testing.assert_allclose(ok[0, 0], k[0, 0], atol=1e-6)
    np.testing.assert_allclose(ov[0, 0], v[0, 0], atol=1e-6)
    # and a plain target RoPE gives plain-rotated keys of the un-rotated source
    gp = synth.ModelGeom(1, 1, 64, 5e5)
    p2 = oracle.OracleProblem(g, gp, [0], [S], [0, S], S, S, [k], [v], W, W)
    ok2, _ = p2.translate()
    for t in (0, 7, 39):
        raw = oracle.rope_g(k[0, 0, t], g, t, -1)
        np.testing.assert_allclose(ok2[0, 0, t], oracle.rope(raw, 5e5, t, +1), atol=1e-6)


# ------------------------------------------------------- partial rotary heads
def test_partial_rotary_over_the_whole_head_is_the_plain_map():
    rng = np.random.default_rng(31)
    x = rng.standard_normal(128)
    for kw in ({}, dict(rope_type=synth.ROPE_LINEAR, rope_factor=4.0)):
        full = oracle.rope_g(x, synth.ModelGeom(1, 1, 128, 1e4, **kw), 321.0, +1)
        same = oracle.rope_g(x, synth.ModelGeom(1, 1, 128, 1e4, rotary_dim=128, **kw), 321.0, +1)
        np.testing.assert_array_equal(full, same)


def test_partial_rotary_is_a_plain_head_of_the_rotated_width_and_passes_the_rest():
    # A head of d channels rotating its first n: the first n channels are the plain map of an
    # n-channel head (pairs (i, i + n/2), frequencies over n), the others are untouched.
    rng = np.random.default_rng(32)
    for d, n in ((128, 32), (128, 64), (128, 96), (256, 64), (64, 16)):
        x = rng.standard_normal(d)
        for kw in ({}, dict(rope_type=synth.ROPE_LINEAR, rope_factor=8.0)):
            gp = synth.ModelGeom(1, 1, d, 1e4, rotary_dim=n, **kw)
            gn = synth.ModelGeom(1, 1, n, 1e4, **kw)
            for pos in (0.0, 5.0, 4095.0):
                y = oracle.rope_g(x, gp, pos, +1)
                np.testing.assert_array_equal(y[:n], oracle.rope_g(x[:n], gn, pos, +1))
                np.testing.assert_array_equal(y[n:], x[n:])
                np.testing.assert_allclose(oracle.rope_g(y, gp, pos, -1), x, atol=1e-12)


def test_partial_rotary_pairs_and_frequency_closed_form():
    # d = 96 with 24 rotated channels (a quarter of the head): channel 1 pairs with channel 13
    # (1 + 24/2, not 1 + 96/2) and turns by theta_1 = base^(-2/24); at position base^(1/12)
    # the angle is exactly 1 rad.
    g = synth.ModelGeom(1, 1, 96, 1e4, rotary_dim=24)
    x = np.zeros(96)
    x[1] = 1.0
    y = oracle.rope_g(x, g, 1e4 ** (1.0 / 12.0), +1)
    want = np.zeros(96)
    want[1], want[13] = np.cos(1.0), np.sin(1.0)
    np.testing.assert_allclose(y, want, atol=1e-13)


def test_partial_rotary_translation_round_trip_and_mixed_heads():
    # Same partial-rotary geometry on both sides, W = I, identity alignment: the stored keys come
    # back.  A fully rotating target instead gets the plain rotation of the un-rotated keys.
    rng = np.random.default_rng(33)
    g = synth.ModelGeom(1, 1, 128, 1e4, rotary_dim=64)
    S = 29
    k = oracle.rope_cache(rng.standard_normal((1, 1, S, 128)).astype(np.float32), g)
    v = rng.standard_normal((1, 1, S, 128)).astype(np.float32)
    W = np.eye(128, dtype=np.float32)[None, None]
    ok, ov = oracle.OracleProblem(g, g, [0], [S], [0, S], S, S, [k], [v], W, W).translate()
    np.testing.assert_allclose(ok[0, 0], k[0, 0], atol=1e-6)
    np.testing.assert_array_equal(ov[0, 0], v[0, 0])
    gf = synth.ModelGeom(1, 1, 128, 1e6)
    ok2, _ = oracle.OracleProblem(g, gf, [0], [S], [0, S], S, S, [k], [v], W, W).translate()
    for t in (0, 9, 28):
        raw = oracle.rope_g(k[0, 0, t].astype(np.float64), g, t, -1)
        np.testing.assert_array_equal(raw[64:], k[0, 0, t, 64:])          # the tail never rotated
        np.testing.assert_allclose(ok2[0, 0, t], oracle.rope(raw, 1e6, t, +1), atol=1e-6)


# ------------------------------------------------------------ translation
def _geom(L, H, d, base):
    return synth.ModelGeom(L, H, d, base)


def _problem(sg, dg, layer_map, lens_src, lens_tgt, src_k, src_v, wk, wv, lo=None, hi=None, sp=None, tp=None):
    so = np.concatenate([[0], np.cumsum(lens_tgt)]).astype(np.int32)
    return oracle.OracleProblem(sg, dg, layer_map, np.array(lens_src, np.int32), so,
                                src_k[0].shape[2], max(lens_tgt), src_k, src_v, wk, wv, lo, hi, sp, tp)


def _rand_src(rng, g, B, S):
    return ([rng.standard_normal((B, g.num_kv_heads, S, g.head_dim)).astype(np.float32) for _ in range(g.num_layers)],
            [rng.standard_normal((B, g.num_kv_heads, S, g.head_dim)).astype(np.float32) for _ in range(g.num_layers)])


def test_identity_translator_round_trip():
    """Same geometry, same tokenizer, W = I: output equals the stored cache."""
    rng = np.random.default_rng(1)
    g = _geom(3, 2, 64, 1e4)
    B, S = 2, 37
    ks, vs = _rand_src(rng, g, B, S)
    ks = [oracle.rope_cache(k, g.rope_base) for k in ks]
    eye = np.broadcast_to(np.eye(64, dtype=np.float32), (3, 2, 64, 64)).copy()
    p = _problem(g, g, [0, 1, 2], [S, S], [S, S], ks, vs, eye, eye)
    ok, ov = p.translate()
    for j in range(3):
        for b in range(B):
            np.testing.assert_allclose(ok[j, :, b * S:(b + 1) * S], ks[j][b], atol=2e-6)
            np.testing.assert_array_equal(ov[j, :, b * S:(b + 1) * S], vs[j][b])


def test_selection_matrix_picks_first_grouped_head():
    """H_s = 2 H_t and W = [I; 0]: target head j reproduces source head 2j."""
    rng = np.random.default_rng(2)
    sg, dg = _geom(2, 4, 64, 1e6), _geom(2, 2, 64, 1e6)
    S = 19
    ks, vs = _rand_src(rng, sg, 1, S)
    ks = [oracle.rope_cache(k, sg.rope_base) for k in ks]
    sel = np.zeros((2, 2, 128, 64), np.float32)
    sel[:, :, :64, :] = np.eye(64)
    p = _problem(sg, dg, [1, 0], [S], [S], ks, vs, sel, sel)
    ok, ov = p.translate()
    for j, l in ((0, 1), (1, 0)):
        for h in range(2):
            np.testing.assert_allclose(ok[j, h], ks[l][0, 2 * h], atol=2e-6)
            np.testing.assert_array_equal(ov[j, h], vs[l][0, 2 * h])
    sel2 = np.zeros_like(sel)
    sel2[:, :, 64:, :] = np.eye(64)      # second half selects head 2j+1
    ok, ov = _problem(sg, dg, [1, 0], [S], [S], ks, vs, sel2, sel2).translate()
    np.testing.assert_array_equal(ov[0, 1], vs[1][0, 3])


def test_expansion_identity_repeats_kv_heads():
    rng = np.random.default_rng(3)
    sg, dg = _geom(1, 2, 64, 1e4), _geom(1, 4, 64, 1e4)
    ks, vs = _rand_src(rng, sg, 1, 11)
    ks = [oracle.rope_cache(k, sg.rope_base) for k in ks]
    eye = np.broadcast_to(np.eye(64, dtype=np.float32), (1, 4, 64, 64)).copy()
    ok, ov = _problem(sg, dg, [0], [11], [11], ks, vs, eye, eye).translate()
    for h in range(4):
        np.testing.assert_allclose(ok[0, h], ks[0][0, h // 2], atol=2e-6)
        np.testing.assert_array_equal(ov[0, h], vs[0][0, h // 2])


def test_no_rope_projection_is_a_matmul_of_the_concatenated_heads():
    """Bases <= 0 and identity alignment reduce the operator to concat(heads) @ W."""
    rng = np.random.default_rng(4)
    sg, dg = _geom(2, 4, 64, 0.0), _geom(2, 2, 128, 0.0)
    S = 9
    ks, vs = _rand_src(rng, sg, 1, S)
    wk = rng.standard_normal((2, 2, 128, 128)).astype(np.float32)
    wv = rng.standard_normal((2, 2, 128, 128)).astype(np.float32)
    ok, ov = _problem(sg, dg, [0, 1], [S], [S], ks, vs, wk, wv).translate()
    for j in range(2):
        for h in range(2):
            xk = np.concatenate([ks[j][0, 2 * h], ks[j][0, 2 * h + 1]], axis=1).astype(np.float64)
            xv = np.concatenate([vs[j][0, 2 * h], vs[j][0, 2 * h + 1]], axis=1).astype(np.float64)
            np.testing.assert_allclose(ok[j, h], xk @ wk[j, h].astype(np.float64), rtol=1e-12, atol=1e-12)
            np.testing.assert_allclose(ov[j, h], xv @ wv[j, h].astype(np.float64), rtol=1e-12, atol=1e-12)


def test_span_closed_form_unrotates_before_the_mean():
    """If every source token of span t stores R(p_s) u_t, the output is R(p_t) W u_t.

    Also V: rows c_s * v_t reduce to mean(c) * W v_t.  Differing source and
    target bases and head dims, cross-tokenizer spans of length 1-3.
    """
    rng = np.random.default_rng(5)
    sg, dg = _geom(1, 2, 64, 1e6), _geom(1, 1, 128, 1e4)
    T = 40
    lo, hi, S, _, _ = synth.draw_spans(T, 9)
    u = rng.standard_normal((T, 2, 64))
    v = rng.standard_normal((T, 2, 64))
    c = rng.uniform(0.5, 2.0, S)
    k_store = np.zeros((1, 2, S, 64), np.float32)
    v_store = np.zeros((1, 2, S, 64), np.float32)
    for t in range(T):
        for s in range(lo[t], hi[t]):
            for g in range(2):
                k_store[0, g, s] = oracle.rope(u[t, g], sg.rope_base, s, +1)
                v_store[0, g, s] = c[s] * v[t, g]
    w = rng.standard_normal((1, 1, 128, 128)).astype(np.float32)
    p = _problem(sg, dg, [0], [S], [T], [k_store], [v_store], w, w, lo, hi)
    ok, ov = p.translate()
    W = w[0, 0].astype(np.float64)
    for t in range(T):
        uk = np.concatenate([k_store[0, 0, lo[t]], k_store[0, 1, lo[t]]]).astype(np.float64)
        uk = np.concatenate([oracle.rope(uk[:64], sg.rope_base, lo[t], -1), oracle.rope(uk[64:], sg.rope_base, lo[t], -1)])
        want_k = oracle.rope(uk @ W, dg.rope_base, t, +1)
        np.testing.assert_allclose(ok[0, 0, t], want_k, atol=1e-5)
        vt = np.concatenate([v[t, 0], v[t, 1]]).astype(np.float32).astype(np.float64)
        want_v = np.mean(c[lo[t]:hi[t]]) * (vt @ W)
        np.testing.assert_allclose(ov[0, 0, t], want_v, rtol=1e-5, atol=1e-5)


def test_linearity_and_batch_invariance():
    rng = np.random.default_rng(6)
    sg, dg = _geom(2, 2, 64, 1e4), _geom(1, 2, 64, 1e6)
    lens = [13, 29]
    S = 29
    k1, v1 = [[synth.bf16_round(x) for x in y] for y in _rand_src(rng, sg, 2, S)]
    k2, v2 = [[synth.bf16_round(x) for x in y] for y in _rand_src(rng, sg, 2, S)]
    w = rng.standard_normal((1, 2, 64, 64)).astype(np.float32)
    a, b = 0.5, -2.0
    km = [a * x + b * y for x, y in zip(k1, k2)]
    vm = [a * x + b * y for x, y in zip(v1, v2)]
    o1 = _problem(sg, dg, [1], lens, lens, k1, v1, w, w).translate()
    o2 = _problem(sg, dg, [1], lens, lens, k2, v2, w, w).translate()
    om = _problem(sg, dg, [1], lens, lens, km, vm, w, w).translate()
    # inputs are bf16-valued, so a*x + b*y is exact in float32 unless the
    # exponents are far apart; the tolerance covers that last rounding
    for i in range(2):
        np.testing.assert_allclose(om[i], a * o1[i] + b * o2[i], rtol=1e-6, atol=2e-5)
    # batch invariance: sequence 1 alone gives the same rows
    solo = _problem(sg, dg, [1], [29], [29], [k[1:2] for k in k1], [v[1:2] for v in v1], w, w).translate()
    for i in range(2):
        np.testing.assert_array_equal(o1[i][:, :, 13:], solo[i])


def test_layer_map_is_followed():
    rng = np.random.default_rng(7)
    sg, dg = _geom(3, 2, 64, 1e4), _geom(2, 2, 64, 1e4)
    ks, vs = _rand_src(rng, sg, 1, 5)
    w = rng.standard_normal((2, 2, 64, 64)).astype(np.float32)
    base = _problem(sg, dg, [2, 0], [5], [5], ks, vs, w, w).translate()
    perm = [ks[2], ks[0], ks[1]], [vs[2], vs[0], vs[1]]
    moved = _problem(sg, dg, [0, 1], [5], [5], perm[0], perm[1], w, w).translate()
    for i in range(2):
        np.testing.assert_array_equal(base[i], moved[i])


# ----------------------------------------------- richer translator forms (Section 5)
def _problem_f(sg, dg, layer_map, lens, src_k, src_v, wk, wv, lo=None, hi=None, **kw):
    so = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    S = src_k[0].shape[2]
    lens_src = [S] * len(lens) if lo is not None else lens
    return oracle.OracleProblem(sg, dg, layer_map, np.array(lens_src, np.int32), so, S, max(lens), src_k, src_v,
                                wk, wv, lo, hi, **kw)


def test_dense_form_without_rope_is_a_matmul_of_all_source_heads():
    """Per-layer form: every target head reads concat(all source heads) @ W[j, h]."""
    rng = np.random.default_rng(31)
    sg, dg = _geom(2, 4, 64, 0.0), _geom(2, 2, 128, 0.0)
    S = 7
    ks, vs = _rand_src(rng, sg, 1, S)
    wk = rng.standard_normal((2, 2, 256, 128)).astype(np.float32)
    wv = rng.standard_normal((2, 2, 256, 128)).astype(np.float32)
    ok, ov = _problem_f(sg, dg, [1, 0], [S], ks, vs, wk, wv, form=1).translate()
    for j, l in ((0, 1), (1, 0)):
        xk = np.concatenate([ks[l][0, g] for g in range(4)], axis=1).astype(np.float64)
        xv = np.concatenate([vs[l][0, g] for g in range(4)], axis=1).astype(np.float64)
        for h in range(2):
            np.testing.assert_allclose(ok[j, h], xk @ wk[j, h].astype(np.float64), rtol=1e-12, atol=1e-12)
            np.testing.assert_allclose(ov[j, h], xv @ wv[j, h].astype(np.float64), rtol=1e-12, atol=1e-12)


def test_dense_form_restricted_to_the_group_equals_the_grouped_form():
    """A dense W that is zero outside target head h's GQA rows gives the grouped result
    (with RoPE on both sides and cross-tokenizer spans)."""
    rng = np.random.default_rng(32)
    sg, dg = _geom(1, 4, 64, 1e6), _geom(1, 2, 64, 1e4)
    T = 25
    lo, hi, S, _, _ = synth.draw_spans(T, 3)
    ks, vs = _rand_src(rng, sg, 1, S)
    ks = [oracle.rope_cache(k, sg.rope_base) for k in ks]
    wg = rng.standard_normal((1, 2, 128, 64)).astype(np.float32)
    wd = np.zeros((1, 2, 256, 64), np.float32)
    for h in range(2):
        wd[0, h, 128 * h:128 * h + 128] = wg[0, h]
    grouped = _problem_f(sg, dg, [0], [T], ks, vs, wg, wg, lo, hi).translate()
    dense = _problem_f(sg, dg, [0], [T], ks, vs, wd, wd, lo, hi, form=1).translate()
    for i in range(2):
        np.testing.assert_allclose(dense[i], grouped[i], rtol=1e-12, atol=1e-12)


def test_layer_groups_concatenate_source_layers():
    """k = 2 source layers per target layer: without RoPE the input is the concatenation of
    both layers' grouped heads; with RoPE and spans, W = [W1; 0] and [0; W2] select one layer
    each and their sum is linear."""
    rng = np.random.default_rng(33)
    sg, dg = _geom(3, 2, 64, 0.0), _geom(1, 1, 64, 0.0)
    S = 6
    ks, vs = _rand_src(rng, sg, 1, S)
    w = rng.standard_normal((1, 1, 256, 64)).astype(np.float32)
    ok, ov = _problem_f(sg, dg, [[2, 0]], [S], ks, vs, w, w, k_layers=2).translate()
    x = np.concatenate([ks[2][0, 0], ks[2][0, 1], ks[0][0, 0], ks[0][0, 1]], axis=1).astype(np.float64)
    np.testing.assert_allclose(ok[0, 0], x @ w[0, 0].astype(np.float64), rtol=1e-12, atol=1e-12)
    # with RoPE and spans
    sg, dg = _geom(3, 2, 64, 1e4), _geom(1, 1, 64, 1e6)
    T = 21
    lo, hi, S, _, _ = synth.draw_spans(T, 4)
    ks, vs = _rand_src(rng, sg, 1, S)
    ks = [oracle.rope_cache(k, sg.rope_base) for k in ks]
    w1 = rng.standard_normal((1, 1, 128, 64)).astype(np.float32)
    w2 = rng.standard_normal((1, 1, 128, 64)).astype(np.float32)
    z = np.zeros_like(w1)
    both = _problem_f(sg, dg, [[2, 1]], [T], ks, vs, np.concatenate([w1, w2], 2), np.concatenate([w1, w2], 2),
                      lo, hi, k_layers=2).translate()
    first = _problem_f(sg, dg, [[2, 1]], [T], ks, vs, np.concatenate([w1, z], 2), np.concatenate([w1, z], 2),
                       lo, hi, k_layers=2).translate()
    only2 = _problem_f(sg, dg, [2], [T], ks, vs, w1, w1, lo, hi).translate()
    only1 = _problem_f(sg, dg, [1], [T], ks, vs, w2, w2, lo, hi).translate()
    for i in range(2):
        np.testing.assert_allclose(first[i], only2[i], rtol=1e-12, atol=1e-12)
        np.testing.assert_allclose(both[i], only2[i] + only1[i], rtol=1e-9, atol=1e-9)


def test_latent_adapter_equals_the_product_matrix():
    """(x A) B = x (A B): the chained maps match a full-rank translator with W = A B, and a
    rank-one adapter gives (x . a) b."""
    rng = np.random.default_rng(34)
    sg, dg = _geom(2, 4, 64, 1e6), _geom(2, 2, 128, 1e4)
    T = 17
    lo, hi, S, _, _ = synth.draw_spans(T, 5)
    ks, vs = _rand_src(rng, sg, 1, S)
    ks = [oracle.rope_cache(k, sg.rope_base) for k in ks]
    for r in (1, 16):
        A = [rng.standard_normal((2, 2, 128, r)).astype(np.float32) for _ in range(2)]
        B = [rng.standard_normal((2, 2, r, 128)).astype(np.float32) for _ in range(2)]
        lr = _problem_f(sg, dg, [1, 0], [T], ks, vs, None, None, lo, hi,
                        low_rank=(A[0], B[0], A[1], B[1])).translate()
        # the product in float64 is not float32-exact: compare with a float64-weight reference
        Wk = np.einsum("jhir,jhro->jhio", A[0].astype(np.float64), B[0].astype(np.float64))
        Wv = np.einsum("jhir,jhro->jhio", A[1].astype(np.float64), B[1].astype(np.float64))
        full = _problem_f(sg, dg, [1, 0], [T], ks, vs, Wk.astype(np.float32), Wv.astype(np.float32),
                          lo, hi).translate()
        for i in range(2):
            scale = np.abs(full[i]).max()
            np.testing.assert_allclose(lr[i], full[i], rtol=0, atol=1e-6 * scale)
    # rank one, V path without RoPE: y = (xbar . a) b
    a, b = A[1][..., :1], B[1][:, :, :1, :]
    _, ov = _problem_f(sg, dg, [1, 0], [T], ks, vs, None, None, lo, hi, low_rank=(a, b, a, b)).translate()
    t = 3
    xbar = np.concatenate([vs[1][0, g, lo[t]:hi[t]].astype(np.float64).mean(0) for g in (0, 1)])
    np.testing.assert_allclose(ov[0, 0, t], (xbar @ a[0, 0, :, 0].astype(np.float64)) * b[0, 0, 0].astype(np.float64),
                               rtol=1e-12, atol=1e-12)


# ------------------------------------------------ closed-form translator fit (Section 5, L_KV)
def _fit_case(rng, sg, dg, layer_map, T, spans_key=None):
    if spans_key is None:
        lo = hi = None
        S = T
    else:
        lo, hi, S, _, _ = synth.draw_spans(T, spans_key)
    ks, vs = _rand_src(rng, sg, 1, S)
    if sg.rope_base > 0:
        ks = [oracle.rope_cache(k, sg.rope_base) for k in ks]
    return ks, vs, lo, hi, S


def test_fit_matches_numpy_least_squares_without_rope():
    """No RoPE, identity alignment: x_t is concat(grouped heads) of row t, y_t the target row;
    the oracle's W equals numpy's least-squares / ridge solutions on X built here from the raw
    arrays."""
    rng = np.random.default_rng(41)
    sg, dg = _geom(2, 4, 64, 0.0), _geom(1, 2, 64, 0.0)
    T = 300
    ks, vs, _, _, S = _fit_case(rng, sg, dg, [1], T)
    tk = [rng.standard_normal((1, 2, T, 64)).astype(np.float32)]
    tv = [rng.standard_normal((1, 2, T, 64)).astype(np.float32)]
    p = _problem_f(sg, dg, [1], [T], ks, vs, np.zeros((1, 2, 128, 64), np.float32),
                   np.zeros((1, 2, 128, 64), np.float32))
    for lam in (0.0, 3.5):
        wk, wv = p.fit(tk, tv, lam)
        for h in range(2):
            for src, tgt, w in ((ks, tk, wk), (vs, tv, wv)):
                X = np.concatenate([src[1][0, 2 * h], src[1][0, 2 * h + 1]], axis=1).astype(np.float64)
                Y = tgt[0][0, h].astype(np.float64)
                if lam == 0.0:
                    ref = np.linalg.lstsq(X, Y, rcond=None)[0]
                else:
                    ref = np.linalg.solve(X.T @ X + lam * np.eye(128), X.T @ Y)
                np.testing.assert_allclose(w[0, h], ref, rtol=1e-9, atol=1e-10)
                # stationarity of the ridge objective
                grad = X.T @ (X @ w[0, h] - Y) + lam * w[0, h]
                assert np.abs(grad).max() < 1e-8 * max(1.0, np.abs(X.T @ Y).max())


def test_fit_recovers_a_planted_translator():
    """Target caches produced by translating with W_true (RoPE on both sides, spans, GQA):
    the un-regularised fit recovers W_true."""
    rng = np.random.default_rng(42)
    sg, dg = _geom(3, 4, 64, 1e6), _geom(2, 2, 64, 1e4)
    T = 400
    ks, vs, lo, hi, S = _fit_case(rng, sg, dg, [2, 0], T, spans_key=7)
    w_true_k = rng.standard_normal((2, 2, 128, 64)).astype(np.float32)
    w_true_v = rng.standard_normal((2, 2, 128, 64)).astype(np.float32)
    p = _problem_f(sg, dg, [2, 0], [T], ks, vs, w_true_k, w_true_v, lo, hi)
    ok, ov = p.translate()                                    # [Lt, Ht, T, dt]
    tk = [ok[j][None].astype(np.float32) for j in range(2)]   # [1, Ht, T, dt]
    tv = [ov[j][None].astype(np.float32) for j in range(2)]
    wk, wv = p.fit(tk, tv, 0.0)
    # the targets were rounded to float32, so recovery is to ~1e-5 relative
    np.testing.assert_allclose(wk, w_true_k, atol=2e-4)
    np.testing.assert_allclose(wv, w_true_v, atol=2e-4)


def test_fit_ridge_shrinks_toward_xty_over_lambda():
    """As lambda grows, lambda W tends to X^T Y."""
    rng = np.random.default_rng(43)
    sg, dg = _geom(1, 1, 64, 1e4), _geom(1, 1, 64, 1e4)
    T = 50
    ks, vs, _, _, S = _fit_case(rng, sg, dg, [0], T)
    tk = [rng.standard_normal((1, 1, T, 64)).astype(np.float32)]
    tv = [rng.standard_normal((1, 1, T, 64)).astype(np.float32)]
    z = np.zeros((1, 1, 64, 64), np.float32)
    p = _problem_f(sg, dg, [0], [T], ks, vs, z, z)
    lam = 1e9
    _, wv = p.fit(tk, tv, lam)
    X = vs[0][0, 0].astype(np.float64)
    np.testing.assert_allclose(lam * wv[0, 0], X.T @ tv[0][0, 0].astype(np.float64), rtol=1e-6, atol=1e-6)
