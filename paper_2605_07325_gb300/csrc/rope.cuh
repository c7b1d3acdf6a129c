// rope.cuh -- the rotation of a query/key pair at an absolute position, shared
// by every kernel that applies it (the RoPE/append kernel and the fused
// foreground attention kernel), so that keys rotated by either are bitwise
// identical.
//
// Element i of a head pairs with element i + d/2 (rotate-half) and turns by
// theta_i = pos * base^(-2i/d).  The turn count pos * base^(-2i/d) / (2 pi) can
// exceed 2^14 at positions past 10^5, where one fp32 ulp of it is already
// 2^-10 turns; it is therefore formed in two fp32 words.  The host splits
// w_i = base^(-2i/d) / (2 pi) (computed in fp64) into w_hi = fl32(w_i) and
// w_lo = fl32(w_i - w_hi); the product pos * w_hi is taken exactly as p + e
// with the fused multiply-add (Dekker's product as TwoProduct-by-FMA: p =
// fl(pos * w_hi), e = fma(pos, w_hi, -p), exact because pos < 2^24 is an
// fp32 integer), the integer part of p is dropped exactly, and the small
// terms e + pos * w_lo are added to the fractional part.  The reduced turn
// count in [-1/2, 1/2] carries an absolute error of a few 2^-25, as one fp32
// rounding of the angle itself would.  Every operation is an explicitly
// rounded intrinsic so no call site contracts it differently.
#pragma once

#include <cstdint>
#include <cuda_bf16.h>

#include "internal.h"

namespace csr {

// Reduced turn count of position pos (< 2^24) for the split frequency w.
// The position is converted from 32 bits: a 64-bit integer conversion costs
// several times the rest of the angle on this GPU.
__device__ __forceinline__ float rope_turns(int64_t pos, TurnSplit w) {
  const float x = __int2float_rn(static_cast<int32_t>(pos));   // exact below 2^24
  const float p = __fmul_rn(x, w.hi);
  const float e = __fmaf_rn(x, w.hi, -p);           // x * w.hi = p + e exactly
  const float frac = __fsub_rn(p, rintf(p));        // exact: p and its nearest integer
  const float small = __fmaf_rn(x, w.lo, e);
  const float t = __fadd_rn(frac, small);
  return __fsub_rn(t, rintf(t));                    // back into [-1/2, 1/2]
}

// cos and sin of 2 pi * turns.
__device__ __forceinline__ void rope_cos_sin(int64_t pos, TurnSplit w, float &c, float &s) {
  sincospif(__fmul_rn(2.0f, rope_turns(pos, w)), &s, &c);
}

__device__ __forceinline__ float bf16_lo_f(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi_f(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }
__device__ __forceinline__ uint32_t pack_bf16x2_rn(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t *>(&v);
}

// Rotate 8 pairs (x[i0..i0+7], x[i0+d/2..i0+d/2+7]) held as two 16-byte
// vectors: x' = x cos - z sin, z' = z cos + x sin, each product rounded, then
// the sum, then the bf16 result (round to nearest even).
__device__ __forceinline__ void rope_rotate8(const uint4 &a, const uint4 &b, const float *cs,
                                             const float *sn, uint4 &ya, uint4 &yb) {
  const uint32_t aw[4] = {a.x, a.y, a.z, a.w};
  const uint32_t bw[4] = {b.x, b.y, b.z, b.w};
  uint32_t ra[4], rb[4];
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const float x0 = bf16_lo_f(aw[e]), x1 = bf16_hi_f(aw[e]);
    const float z0 = bf16_lo_f(bw[e]), z1 = bf16_hi_f(bw[e]);
    const float c0 = cs[2 * e], c1 = cs[2 * e + 1];
    const float s0 = sn[2 * e], s1 = sn[2 * e + 1];
    ra[e] = pack_bf16x2_rn(__fsub_rn(__fmul_rn(x0, c0), __fmul_rn(z0, s0)),
                           __fsub_rn(__fmul_rn(x1, c1), __fmul_rn(z1, s1)));
    rb[e] = pack_bf16x2_rn(__fadd_rn(__fmul_rn(z0, c0), __fmul_rn(x0, s0)),
                           __fadd_rn(__fmul_rn(z1, c1), __fmul_rn(x1, s1)));
  }
  ya = make_uint4(ra[0], ra[1], ra[2], ra[3]);
  yb = make_uint4(rb[0], rb[1], rb[2], rb[3]);
}

}  // namespace csr
