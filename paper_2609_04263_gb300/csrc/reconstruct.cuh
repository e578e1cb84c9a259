// Reconstruction of stored keys/values for the prefill attention kernels
// (attend_prefill_mma.cu): the value the cache stores
// for a token and channel, per format (Section 3.1): codes x scale + offset
// for the quantized formats, the full-precision copy for FLOAT caches and
// the KIVI residual window.
#pragma once

#include "kvq_internal.cuh"

namespace kvq {

// Reconstruct channels 8c .. 8c+7 of token t (keys: which = 0) in fp32.
__device__ __forceinline__ void deq8(const Geom& g, int which, int b, int h, int t, int c,
                                     int T, int tq, float v[8]) {
  if (t >= T) {
#pragma unroll
    for (int e = 0; e < 8; ++e) v[e] = 0.f;
    return;
  }
  const int G = g.G, bits = which ? g.vb : g.kb;
  const int P_CODES = which ? KVQ_PLANE_V_CODES : KVQ_PLANE_K_CODES;
  const int P_SCALE = which ? KVQ_PLANE_V_SCALE : KVQ_PLANE_K_SCALE;
  const int P_ZERO = which ? KVQ_PLANE_V_ZERO : KVQ_PLANE_K_ZERO;
  const int P_FULL = which ? KVQ_PLANE_V_FULL : KVQ_PLANE_K_FULL;
  const bool raw = g.fmt == KVQ_FMT_FLOAT || (g.fmt == KVQ_FMT_KIVI && t >= tq);
  if (raw) {
    const int slot = g.fmt == KVQ_FMT_KIVI ? t % g.ring : t;
    const uint4 u = *reinterpret_cast<const uint4*>(
        plane_ptr<__nv_bfloat16>(g, P_FULL, b, h, slot, 8 * c));
    const __nv_bfloat16* e8 = reinterpret_cast<const __nv_bfloat16*>(&u);
#pragma unroll
    for (int e = 0; e < 8; ++e) v[e] = __bfloat162float(e8[e]);
    return;
  }
  const uint8_t* row = plane_ptr<uint8_t>(g, P_CODES, b, h, t);
  uint64_t w;
  if (bits == 4) w = *reinterpret_cast<const uint32_t*>(row + 4 * c);
  else if (bits == 2) w = *reinterpret_cast<const uint16_t*>(row + 2 * c);
  else w = *reinterpret_cast<const uint64_t*>(row + 8 * c);
  const unsigned mask = (1u << bits) - 1;
  if (g.fmt == KVQ_FMT_KIVI && which == 0) {   // per channel: scale and zero per (block, d)
    const uint4 su = *reinterpret_cast<const uint4*>(
        plane_ptr<__half>(g, KVQ_PLANE_K_SCALE, b, h, t / G, 8 * c));
    const uint4 zu = *reinterpret_cast<const uint4*>(
        plane_ptr<__half>(g, KVQ_PLANE_K_ZERO, b, h, t / G, 8 * c));
    const __half* s8 = reinterpret_cast<const __half*>(&su);
    const __half* z8 = reinterpret_cast<const __half*>(&zu);
#pragma unroll
    for (int e = 0; e < 8; ++e)
      v[e] = (float)((w >> (e * bits)) & mask) * __half2float(s8[e]) + __half2float(z8[e]);
  } else {
    const int grp = (8 * c) / G;
    const float s = __half2float(*plane_ptr<__half>(g, P_SCALE, b, h, t, grp));
    float m;
    if (g.fmt == KVQ_FMT_SYMMETRIC) m = -(float)(1 << (bits - 1)) * s;
    else m = __half2float(*plane_ptr<__half>(g, P_ZERO, b, h, t, grp));
#pragma unroll
    for (int e = 0; e < 8; ++e) v[e] = (float)((w >> (e * bits)) & mask) * s + m;
  }
}


}  // namespace kvq
