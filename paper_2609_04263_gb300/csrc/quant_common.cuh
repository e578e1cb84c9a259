// Grouped quantizer arithmetic shared by the kernels that code keys and
// values into the cache (pack.cu; the projection epilogue of project_tc.cu
// when it appends): every value that decides a code is computed in IEEE fp32
// with explicitly rounded operations, in the order the cache format fixes
// (Section 3.1, Eq. (affine) and the symmetric control), so every writer
// produces the same codes and fp16 metadata bit for bit.
#pragma once

#include "kvq_internal.cuh"

namespace kvq {
namespace quant {

// Eq. (affine) scale for one group: max((mx - mn) / (2^b - 1), 1e-8).
__device__ __forceinline__ float affine_scale(float mn, float mx, int bits) {
  return fmaxf(__fdiv_rn(__fsub_rn(mx, mn), (float)((1 << bits) - 1)), 1e-8f);
}
// rint(a / s) where the quotient is first rounded to fp32 (both roundings to
// nearest even), which is how the cache format defines a code.  inv is the
// correctly rounded reciprocal of s (one per group), so q = RN(a inv) is
// within 2^-23 |a / s| of a / s, below 2^-17 for |q| < 64.  When q lies
// farther than 2^-14 from the half-integer between its two neighbouring
// integers, the exact quotient and its fp32 rounding lie on the same side of
// that representable half-integer (rounding is monotone), so all three round
// to the same integer.  Otherwise (near a tie, or NaN / out of range) the IEEE
// quotient is formed.
__device__ __forceinline__ float rint_quot(float a, float s, float inv) {
  const float q = __fmul_rn(a, inv);
  const float d = fabsf(q - (floorf(q) + 0.5f));
  if (d > 0x1p-14f && fabsf(q) < 64.f) return rintf(q);
  return rintf(__fdiv_rn(a, s));
}
// The fast half of rint_quot without a branch: ok is cleared when the
// caller must form the IEEE quotient instead (loops then redo their
// elements once, exactly, when any was near a tie).
__device__ __forceinline__ float rint_quot_fast(float a, float inv, bool& ok) {
  const float q = __fmul_rn(a, inv);
  const float d = fabsf(q - (floorf(q) + 0.5f));
  ok = ok && d > 0x1p-14f && fabsf(q) < 64.f;
  return rintf(q);
}
__device__ __forceinline__ int clamp_code(float c, int bits) {
  return (int)fminf(fmaxf(c, 0.f), (float)((1 << bits) - 1));
}

__device__ __forceinline__ int affine_code(float x, float mn, float s, float inv, int bits) {
  float c = rint_quot(__fsub_rn(x, mn), s, inv);
  c = fminf(fmaxf(c, 0.f), (float)((1 << bits) - 1));
  return (int)c;
}
// Symmetric control: s = max(absmax / qmax, 1e-8), q = round(x / s) in
// [-qmax, qmax], stored as q + 2^(b-1).
__device__ __forceinline__ float sym_scale(float amax, int bits) {
  return fmaxf(__fdiv_rn(amax, (float)((1 << (bits - 1)) - 1)), 1e-8f);
}

// The 8 codes of one lane, LSB first (8 x BITS bits).
template <int BITS, bool SYM>
__device__ __forceinline__ uint64_t code8(const float v[8], float lo, float hi, float* s_out) {
  const float s = SYM ? sym_scale(hi, BITS) : affine_scale(lo, hi, BITS);
  const float inv = __frcp_rn(s);
  *s_out = s;
  constexpr int half = 1 << (BITS - 1);
  bool ok = true;
  float c[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const float a = SYM ? v[i] : __fsub_rn(v[i], lo);
    c[i] = rint_quot_fast(a, inv, ok);
  }
  if (!ok) {
#pragma unroll
    for (int i = 0; i < 8; ++i) c[i] = rintf(__fdiv_rn(SYM ? v[i] : __fsub_rn(v[i], lo), s));
  }
  uint64_t w = 0;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    // the clamps of sym_code / affine_code
    const int code = SYM ? (int)fminf(fmaxf(c[i], (float)(1 - half)), (float)(half - 1)) + half
                         : clamp_code(c[i], BITS);
    w |= (uint64_t)code << (i * BITS);
  }
  return w;
}

// append_arrive with the arrivals spread over 32 counters (words 16..47 of
// the state's padding): the CTAs of bucket id % 32 count themselves, the last
// of each bucket counts the bucket, and the last bucket advances the token
// count, so thousands of CTAs do not queue on one address.
__device__ __forceinline__ void append_arrive_spread(CacheState* st, int T0, int L, bool ok) {
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    constexpr unsigned kBuckets = 32;
    const unsigned total = gridDim.x * gridDim.y * gridDim.z;
    const unsigned id = blockIdx.x + gridDim.x * (blockIdx.y + gridDim.y * blockIdx.z);
    const unsigned nb = total < kBuckets ? total : kBuckets;
    const unsigned b = id % nb;
    const unsigned members = total / nb + (b < total % nb ? 1u : 0u);
    unsigned* bucket = reinterpret_cast<unsigned*>(&st->pad[16 + b]);
    if (atomicAdd(bucket, 1u) == members - 1) {
      *bucket = 0;
      __threadfence();
      if (atomicAdd(&st->done, 1u) == nb - 1) {
        if (ok) st->tokens = T0 + L;
        st->done = 0;
        __threadfence();
      }
    }
  }
}

}  // namespace quant
}  // namespace kvq
