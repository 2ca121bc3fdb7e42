// rope.cuh -- rotary position encoding as the attention uses it (rotate-half
// pairs (i, i + D/2), angle pos * theta^(-2i/D); Sec. 3.2 "Sparse Input
// Construction": retained suffix tokens keep their original positions).  Shared
// by the attention pre-pass and the prefix-cache append, so that a key rotated by
// either lands on the same bf16 value.
#pragma once

#include <cuda_bf16.h>

#include <cmath>
#include <cstdint>

namespace ssm {

__device__ __forceinline__ uint32_t rope_pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&h);
}

// The D/2 rotation frequencies f_i = theta^(-2i/D) (radians per position, formed
// in fp64; all 0 when theta == 0: no rotation), each held as turns per position in
// 0.64 fixed point: turn_i = round(2^64 * f_i / (2 pi)).  A position's angle
// pos * f_i modulo one turn is then the wrapping 64-bit product pos * turn_i,
// exact up to pos units in the last place (< 2^-33 turns for any int32 position),
// with no fp64 arithmetic on the device: GB300's fp64 rate is a small fraction of its fp32 rate, and an
// fp64 range reduction per angle (and an fp64 exponential and logarithm per
// table entry) was a visible part of the pre-pass.  Formed on the host once per
// launch and passed to the kernels by value.
template <int D>
struct RopeFreqs {
  uint64_t turn[D / 2];
};

template <int D>
inline RopeFreqs<D> rope_freqs(float theta) {
  // 1 / (2 pi) as an unevaluated sum of two doubles (about 106 bits)
  constexpr double kInv2PiHi = 0.15915494309189535, kInv2PiLo = -9.839338337591243e-18;
  RopeFreqs<D> r;
  const double l2 = theta > 0.f ? std::log2(static_cast<double>(theta)) : 0.0;
  for (int i = 0; i < D / 2; ++i) {
    if (!(theta > 0.f)) {
      r.turn[i] = 0;
      continue;
    }
    const double f = std::exp2(-(2.0 * i / D) * l2);  // radians per position, <= 1
    // f / (2 pi) in double-double: the product's rounding error recovered with an fma
    const double hi = f * kInv2PiHi;
    const double lo = std::fma(f, kInv2PiHi, -hi) + f * kInv2PiLo;
    // scaled to 2^64 (hi < 0.16, so its scaled value is below 2^62): whole part, then the rest
    const double a = std::ldexp(hi, 64), b = std::ldexp(lo, 64);
    const double af = std::floor(a);
    r.turn[i] = static_cast<uint64_t>(af) + static_cast<uint64_t>(static_cast<int64_t>(std::llrint((a - af) + b)));
  }
  return r;
}

// sin and cos of the angle pos * theta^(-2i/D): its fraction of a turn from the
// wrapping fixed-point product, as a signed 32-bit fraction in [-1/2, 1/2), turned
// into radians in [-pi, pi) in fp32, where sincosf needs no large-argument reduction.
__device__ __forceinline__ void rope_sincos(int32_t pos, uint64_t turn, float& sn, float& cs) {
  const uint64_t t = static_cast<uint64_t>(static_cast<int64_t>(pos)) * turn;
  const int32_t q = static_cast<int32_t>(t >> 32);
  constexpr float kTwoPiOver2p32 = 1.4629180792671596e-09f;  // 2 pi / 2^32
  sincosf(static_cast<float>(q) * kTwoPiOver2p32, &sn, &cs);
}

// Rotates four pairs: x1 holds elements i..i+3 and x2 elements i+D/2..i+D/2+3 of
// one head vector (bf16); y1 = x1 cos - x2 sin, y2 = x2 cos + x1 sin in fp32
// (the product with sin rounded, then one fused multiply-add: the same bits in
// every kernel that includes this), rounded to bf16.
__device__ __forceinline__ void rope_rotate4(uint2 x1, uint2 x2, const float (&cs)[4], const float (&sn)[4],
                                             uint2& y1, uint2& y2) {
  const float a[4] = {__uint_as_float(x1.x << 16), __uint_as_float(x1.x & 0xFFFF0000u),
                      __uint_as_float(x1.y << 16), __uint_as_float(x1.y & 0xFFFF0000u)};
  const float b[4] = {__uint_as_float(x2.x << 16), __uint_as_float(x2.x & 0xFFFF0000u),
                      __uint_as_float(x2.y << 16), __uint_as_float(x2.y & 0xFFFF0000u)};
  float r1[4], r2[4];
#pragma unroll
  for (int t = 0; t < 4; ++t) {
    r1[t] = __fmaf_rn(a[t], cs[t], -__fmul_rn(b[t], sn[t]));
    r2[t] = __fmaf_rn(b[t], cs[t], __fmul_rn(a[t], sn[t]));
  }
  y1 = make_uint2(rope_pack_bf16x2(r1[0], r1[1]), rope_pack_bf16x2(r1[2], r1[3]));
  y2 = make_uint2(rope_pack_bf16x2(r2[0], r2[1]), rope_pack_bf16x2(r2[2], r2[3]));
}

}  // namespace ssm
