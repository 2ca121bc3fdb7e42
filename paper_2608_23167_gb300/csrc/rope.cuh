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

// The D/2 inverse frequencies theta^(-2i/D) in fp64 (all 0 when theta == 0: no
// rotation).  They are formed on the host, once per launch, and passed to the
// kernels by value: GB300's fp64 rate is a small fraction of its fp32 rate, and
// the fp64 exponential and logarithm of every CTA's table were a visible part of
// a small launch.
template <int D>
struct RopeFreqs {
  double f[D / 2];
};

template <int D>
inline RopeFreqs<D> rope_freqs(float theta) {
  RopeFreqs<D> r;
  const double l2 = theta > 0.f ? std::log2(static_cast<double>(theta)) : 0.0;
  for (int i = 0; i < D / 2; ++i) r.f[i] = theta > 0.f ? std::exp2(-(2.0 * i / D) * l2) : 0.0;
  return r;
}

// sin and cos of pos * inv_freq: the angle is formed and reduced modulo 2 pi in
// fp64 (two-part 2 pi), then sin/cos are taken in fp32 on the reduced angle.
__device__ __forceinline__ void rope_sincos(int32_t pos, double inv_freq, float& sn, float& cs) {
  const double a = static_cast<double>(pos) * inv_freq;
  const double k = rint(a * 0.15915494309189535);  // a / (2 pi)
  double r = fma(-k, 6.283185307179586, a);
  r = fma(-k, 2.4492935982947064e-16, r);
  sincosf(static_cast<float>(r), &sn, &cs);
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
