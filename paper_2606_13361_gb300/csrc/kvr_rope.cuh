// kvr_rope.cuh -- the per-head QK-RMSNorm + rotate-half RoPE of the append step,
// shared by every kernel that appends tokens so the cached keys and the roped
// queries are bit-for-bit the same whichever kernel produced them.
//
// Layout: the D/8 threads of one head vector are consecutive lanes of a warp,
// aligned to D/8; thread li (0..D/8-1) holds elements [8*li, 8*li+8).  The sum
// of squares is reduced with xor-shuffles inside that group; the rotate-half
// partner of element i < D/2 (i + D/2) sits in lane li ^ (D/16).  Every product
// and sum is an explicit IEEE fp32 operation (no contraction choices left to
// the compiler), rounded once to bf16 at the end.
#pragma once

#include <stdint.h>

namespace kvr {

__device__ __forceinline__ void bf16x8_to_f32(const uint4& u, float (&x)[8]) {
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    x[2 * i] = __uint_as_float(w[i] << 16);
    x[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
  }
}

__device__ __forceinline__ uint32_t f32x2_to_bf16x2(float lo, float hi) {
  uint32_t r;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

// y = RoPE(RMSNorm(x) * w) for this thread's 8 elements.  `cs` holds the
// (cos, sin) pairs of frequency index (li % (D/16)) * 8 .. +8 for the token's
// position.  All D/8 lanes of the vector must call this together (shuffles).
template <int D>
__device__ __forceinline__ uint4 norm_rope8v(const uint4& xraw, const uint4& wraw, int li, const float2 (&cs)[8],
                                             float eps) {
  constexpr int TPI = D / 8;
  constexpr int HALF_T = TPI / 2;
  float x[8], w[8];
  bf16x8_to_f32(xraw, x);
  bf16x8_to_f32(wraw, w);
  float ss = 0.f;
#pragma unroll
  for (int i = 0; i < 8; ++i) ss = __fmaf_rn(x[i], x[i], ss);
#pragma unroll
  for (int off = TPI / 2; off >= 1; off >>= 1) ss = __fadd_rn(ss, __shfl_xor_sync(0xffffffffu, ss, off, TPI));
  const float inv = __frcp_rn(__fsqrt_rn(__fadd_rn(__fdiv_rn(ss, static_cast<float>(D)), eps)));
  const bool first = li < HALF_T;
  float r[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const float y = __fmul_rn(__fmul_rn(x[i], inv), w[i]);
    const float partner = __shfl_xor_sync(0xffffffffu, y, HALF_T, TPI);
    const float2 e = cs[i];
    const float t = __fmul_rn(partner, e.y);
    r[i] = first ? __fmaf_rn(y, e.x, -t) : __fmaf_rn(y, e.x, t);
  }
  return make_uint4(f32x2_to_bf16x2(r[0], r[1]), f32x2_to_bf16x2(r[2], r[3]), f32x2_to_bf16x2(r[4], r[5]),
                    f32x2_to_bf16x2(r[6], r[7]));
}

// The same, reading this lane's 8 (cos, sin) pairs from the table.
template <int D>
__device__ __forceinline__ uint4 norm_rope8(const uint4& xraw, const uint4& wraw, int li, const float2* cs,
                                            float eps) {
  float2 v[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) v[i] = cs[i];
  return norm_rope8v<D>(xraw, wraw, li, v, eps);
}

}  // namespace kvr
