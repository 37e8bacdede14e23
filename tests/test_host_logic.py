"""Host-side logic of the library's kernel header, checked on the CPU.

A small host program (`host_logic_probe.cu`) is compiled with nvcc against
`paper_2608_30963_gb300/csrc/kvx_common.cuh` and prints what the kernels' index and frequency
helpers compute:
- pair_channels (partial rotary heads): the pair slots cover every channel of a head once,
  rotating slots pair (i, i + n/2), and chunks of 8 slots map to runs of 8 channels;
- rope_inv_freq: the per-pair frequency under each schedule and rotary width equals the angle
  the oracle turns a unit vector by at position 1;
- rope_schedule_ok: the rotary-width rule (0, or a multiple of 16 in [16, head_dim]);
- pair_v_shares (`kvx_schedule.h`): the identity-alignment kernel's V shares form a permutation
  of the CTAs, and under the split's own cost model the costliest CTA costs no more than with
  each CTA taking the mirrored V share.
"""
import os
import shutil
import subprocess

import numpy as np
import pytest

import oracle
from paper_2608_30963_gb300 import synth

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)


@pytest.fixture(scope="module")
def probe(tmp_path_factory):
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(nvcc):
        pytest.skip("nvcc not found")
    exe = str(tmp_path_factory.mktemp("probe") / "host_logic_probe")
    subprocess.check_call([nvcc, "-std=c++17", "-I" + os.path.join(ROOT, "include"),
                           os.path.join(HERE, "host_logic_probe.cu"), "-o", exe])

    def run(lines):
        out = subprocess.run([exe], input="\n".join(lines) + "\n", capture_output=True, text=True, check=True)
        return out.stdout.splitlines()
    return run


@pytest.mark.parametrize("d,n", [(64, 64), (64, 16), (128, 128), (128, 32), (128, 64), (128, 96), (256, 64),
                                 (256, 256), (256, 192)])
def test_pair_slots_cover_every_channel_once(probe, d, n):
    rh = n // 2
    lines = probe([f"pairs {d} {rh}"])
    assert lines[0] == f"pairs {d} {rh}"
    rows = np.array([[int(v) for v in ln.split()] for ln in lines[1:]])
    k, lo, hi = rows[:, 0], rows[:, 1], rows[:, 2]
    assert np.array_equal(np.sort(np.concatenate([lo, hi])), np.arange(d))
    rot = k < rh
    assert np.array_equal(lo[rot], k[rot]) and np.array_equal(hi[rot], k[rot] + rh)
    if n == d:
        assert np.array_equal(hi, lo + d // 2)
    for c in range(0, d // 2, 8):                     # a 16-byte chunk of slots: two runs of 8 channels
        assert np.array_equal(np.diff(lo[c:c + 8]), np.ones(7)) and np.array_equal(np.diff(hi[c:c + 8]), np.ones(7))


SCHED = [
    dict(),
    dict(rope_type=synth.ROPE_LINEAR, rope_factor=4.0),
    dict(rope_type=synth.ROPE_LLAMA3, rope_factor=8.0, rope_low_freq_factor=1.0, rope_high_freq_factor=4.0,
         rope_original_max_position=8192),
]


@pytest.mark.parametrize("d,n,base", [(128, 0, 1e6), (128, 64, 1e4), (64, 32, 1e4), (256, 96, 5e5), (128, 0, 5e5)])
@pytest.mark.parametrize("si", range(len(SCHED)), ids=["plain", "linear", "llama3"])
def test_library_frequencies_equal_the_oracle_angles(probe, d, n, base, si):
    kw = SCHED[si]
    g = synth.ModelGeom(1, 1, d, base, rotary_dim=n, **kw)
    lines = probe([f"freq {d} {n} {g.rope_type} {g.rope_factor} {g.rope_low_freq_factor} "
                   f"{g.rope_high_freq_factor} {g.rope_original_max_position} {base}"])
    h = int(lines[0].split()[1])
    assert h == (n or d) // 2
    f = np.array([float(ln.split()[1]) for ln in lines[1:]])
    # the oracle's angle for pair i at position 1: rotate the unit vector e_i and read the angle
    want = np.empty(h)
    for i in range(h):
        x = np.zeros(d)
        x[i] = 1.0
        y = oracle.rope_g(x, g, 1.0, +1)
        want[i] = np.arctan2(y[i + h], y[i])
    np.testing.assert_allclose(f, want, rtol=1e-12, atol=0)


@pytest.mark.parametrize("d,n,ok", [(128, 0, 1), (128, 16, 1), (128, 128, 1), (128, 112, 1), (128, 24, 0),
                                    (128, 8, 0), (128, 144, 0), (128, -16, 0), (64, 64, 1), (256, 256, 1)])
def test_rotary_width_rule(probe, d, n, ok):
    assert probe([f"ok {d} {n} 0 1 1 4 8192 10000"]) == [f"ok {ok}"]


def _share_cost(r, grid, uh, mt, per_unit):
    a, b = r * uh // grid, (r + 1) * uh // grid
    groups = (b - 1) // mt - a // mt + 1 if b > a else 0
    return per_unit * (b - a) + 0.57 * max(groups - 1, 0)


@pytest.mark.parametrize("grid,uh,mt", [(152, 56 * 32, 32), (152, 56 * 67, 67), (152, 56 * 259, 259), (148, 1000, 9),
                                        (20, 13, 13), (1, 5, 5), (152, 152, 32)])
def test_v_shares_are_a_permutation_that_lowers_the_costliest_cta(probe, grid, uh, mt):
    out = probe([f"vshares {grid} {uh} {mt}"])
    assert out[0] == f"vshares {grid}"
    v = [int(line.split()[1]) for line in out[1:1 + grid]]
    assert sorted(v) == list(range(grid))
    k = [_share_cost(c, grid, uh, mt, 1.41) for c in range(grid)]
    vc = [_share_cost(r, grid, uh, mt, 1.0) for r in range(grid)]
    paired = max(k[c] + vc[v[c]] for c in range(grid))
    mirrored = max(k[c] + vc[grid - 1 - c] for c in range(grid))
    assert paired <= mirrored + 1e-9
