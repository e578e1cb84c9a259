// Pieces shared by the streaming decode kernels (decode_stream.cu for
// affine, symmetric and KIVI caches; decode_stream_kvarn.cu for KVarN): the
// work split, the ring and warp geometry, the merge scratch, and small
// fragment helpers.
#pragma once

#include "decode_attn.cuh"

namespace kvq {
namespace stream {

constexpr int kBT = 32;            // tokens per block (one KIVI key block)
constexpr int kSB = 8;             // blocks per ring stage (copied together)
constexpr int kNW = 11;            // consumer warps (12 warps: the register file holds 168 a thread)
constexpr int kThreads = (kNW + 1) * 32;
constexpr int kMaxStages = 64;
constexpr int kSmemMax = 227 * 1024;
// workspace slot where a KVarN head's coded-token partial waits for the
// combine with the full-precision tokens' split partials (slots below it)
constexpr int kFinalSlot = kMaxSplits - 1;

// Transpose of an 8x8 tile of 16-bit values held as an mma fragment.
__device__ __forceinline__ uint32_t movmatrix_t(uint32_t a) {
  uint32_t d;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(d) : "r"(a));
  return d;
}
__device__ __forceinline__ uint32_t hmul2u(uint32_t a, uint32_t b) {
  __half2 r = __hmul2(*reinterpret_cast<const __half2*>(&a), *reinterpret_cast<const __half2*>(&b));
  return *reinterpret_cast<uint32_t*>(&r);
}
// a * b - c as one fused fp16x2 operation: with c = a * b rounded, the
// exact rounding error of the product
__device__ __forceinline__ uint32_t hfma2u_neg(uint32_t a, uint32_t b, uint32_t c) {
  __half2 r = __hfma2(*reinterpret_cast<const __half2*>(&a), *reinterpret_cast<const __half2*>(&b),
                      __hneg2(*reinterpret_cast<const __half2*>(&c)));
  return *reinterpret_cast<uint32_t*>(&r);
}
__device__ __forceinline__ uint32_t h2u(__half lo, __half hi) {
  return (uint32_t)__half_as_ushort(lo) | ((uint32_t)__half_as_ushort(hi) << 16);
}
__device__ __forceinline__ void mbar_arrive1(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(dattn::smem_u32(bar)) : "memory");
}

// First block index of CTA c when N blocks are cut into P ranges.
__device__ __forceinline__ int64_t range_start(int64_t c, int64_t N, int P) { return c * N / P; }
// The CTA whose range holds block x.
__device__ __forceinline__ int cta_of(int64_t x, int64_t N, int P) {
  int c = (int)(x * P / N);
  while (c + 1 < P && range_start(c + 1, N, P) <= x) ++c;
  while (c > 0 && range_start(c, N, P) > x) --c;
  return c;
}

// Merge scratch after the per-warp partial slots.
struct Merge {
  float m[kMaxSplits][8];   // partials' m (log2 units), then their weights
  float l[kMaxSplits][8];
  float M[8], L[8];
  int last;
  int pad;
};
// Barrier among the consumer warps (the producer warp does not join).
__device__ __forceinline__ void consumer_sync() {
  asm volatile("bar.sync 1, %0;" ::"n"(kNW * 32) : "memory");
}

}  // namespace stream
}  // namespace kvq
