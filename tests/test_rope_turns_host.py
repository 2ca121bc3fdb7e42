"""Host-side check of the RoPE angle table the kernels take (no GPU needed).

The pre-pass and the prefix-cache append form each rotation frequency
f_i = theta^(-2i/d) (radians per position) in fp64 and hold it as turns per
position in 0.64 fixed point, turn_i = round(2^64 * f_i / (2 pi)); a position's
angle modulo one turn is the wrapping 64-bit product pos * turn_i.  This compiles
the table's host code (csrc/rope.cuh) into a small host program and checks it
against the same quantity in 200-bit arithmetic from the same fp64 frequency (the
oracle's frequency carries the same fp64 rounding): every entry within one unit
of 2^-64 turns, so the reduced angle pos * f_i of any int32 position is exact to
below 2^-33 turns; the fp64 frequency itself is within a relative 2^-47 of
theta^(-2i/d) (the rounding of its exponent, scaled by the exponent); and the reduced angles of large positions against pos * f_i
mod 2 pi.
"""
import math
import os
import shutil
import subprocess
import tempfile

import pytest

mpmath = pytest.importorskip("mpmath")

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2608_23167_gb300", "csrc")
INCLUDE = os.path.join(ROOT, "include")

PROGRAM = r"""
#include <cstdio>
#include "rope.cuh"
template <int D> void dump(float theta) {
  const auto r = ssm::rope_freqs<D>(theta);
  for (int i = 0; i < D / 2; ++i) std::printf("%d %.9g %d %llu\n", D, theta, i, (unsigned long long)r.turn[i]);
}
int main() {
  const float thetas[] = {10000.f, 500000.f, 1000000.f, 0.f};
  for (float t : thetas) { dump<64>(t); dump<128>(t); }
  return 0;
}
"""


def _nvcc():
    for c in (os.environ.get("NVCC"), "/usr/local/cuda/bin/nvcc", shutil.which("nvcc")):
        if c and os.path.exists(c):
            return c
    return None


@pytest.fixture(scope="module")
def table():
    nvcc = _nvcc()
    if nvcc is None:
        pytest.skip("nvcc not found")
    with tempfile.TemporaryDirectory() as d:
        src = os.path.join(d, "turns.cu")
        exe = os.path.join(d, "turns")
        with open(src, "w") as f:
            f.write(PROGRAM)
        subprocess.run([nvcc, "-std=c++17", "-I", CSRC, "-I", INCLUDE, src, "-o", exe], check=True,
                       capture_output=True)
        out = subprocess.run([exe], check=True, capture_output=True, text=True).stdout
    rows = []
    for line in out.splitlines():
        d, theta, i, turn = line.split()
        rows.append((int(d), float(theta), int(i), int(turn)))
    return rows


def _freq(theta, i, d):
    """The fp64 frequency as the host forms it: exp2(-(2i/d) * log2(theta))."""
    return math.exp2(-(2.0 * i / d) * math.log2(theta))


def test_turn_table_within_one_unit(table):
    mpmath.mp.prec = 200
    two64 = mpmath.mpf(2) ** 64
    assert len(table) == 4 * (32 + 64)
    for d, theta, i, turn in table:
        assert 0 <= turn < 2 ** 64
        if theta == 0.0:
            assert turn == 0          # theta == 0: no rotation
            continue
        f = _freq(theta, i, d)
        true_f = mpmath.power(mpmath.mpf(theta), mpmath.mpf(-2 * i) / d)
        # exp2 of the rounded exponent (|exponent| < 20): within a few units of 2^-52 relative
        assert abs(mpmath.mpf(f) - true_f) <= true_f * mpmath.mpf(2) ** -47, (d, theta, i)
        exact = mpmath.mpf(f) / (2 * mpmath.pi) * two64
        assert abs(mpmath.mpf(turn) - exact) <= 1, (d, theta, i)
    # i = 0 is one radian per position: 2^64 / (2 pi) turns
    t0 = [t for d, th, i, t in table if i == 0 and th > 0]
    assert all(abs(mpmath.mpf(t) - two64 / (2 * mpmath.pi)) <= 1 for t in t0)


def test_reduced_angles_of_large_positions(table):
    """The kernel's angle: the top 32 bits of (pos * turn_i) mod 2^64 as a signed fraction of a
    turn.  Against pos * theta^(-2i/d) mod 2 pi in 200-bit arithmetic, for positions up to 2^31 - 1."""
    mpmath.mp.prec = 200
    for d, theta, i, turn in table:
        if theta == 0.0 or d != 128 or i % 7:
            continue
        for pos in (0, 1, 3071, 65537, 2 ** 31 - 1):
            t = (pos * turn) % 2 ** 64
            q = (t >> 32) - (1 << 32) * ((t >> 63) & 1)     # signed 32-bit
            got = q * 2 * math.pi / 2 ** 32
            exact = mpmath.fmod(pos * mpmath.mpf(_freq(theta, i, d)), 2 * mpmath.pi)
            if exact >= mpmath.pi:
                exact -= 2 * mpmath.pi
            err = abs(float(exact) - got)
            err = min(err, abs(err - 2 * math.pi))
            # the truncation to 32 bits (2^-32 turn) plus the table's error times pos (< 2^-33 turn)
            assert err <= 2 * math.pi * (2.0 ** -32 + 2.0 ** -33), (theta, i, pos, err)
