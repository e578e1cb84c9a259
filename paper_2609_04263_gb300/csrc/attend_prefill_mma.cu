// Causal prefill attention over the packed cache on tensor cores (bf16
// mma.sync), Sections 3.1-3.3: the L newest queries attend to the stored
// reconstruction of every cached token.
//
// One CTA = (query tile, kv head, sequence).  Its ROWS rows are the g query
// heads of the kv head times nq = ROWS / g consecutive queries, 16 rows per
// warp, so every key/value tile is reconstructed once and shared by all g
// heads.  Per KV tile of NT tokens: the CTA reconstructs K and V into shared
// memory (codes x fp16 scale + fp16 offset; full-precision windows copied):
// K as a bf16 high part plus a bf16 remainder, so that Q K^T (two bf16 MMAs
// per tile) carries about 16 significant bits of K (with real activations the
// logits are large and a bf16-rounded K would move them visibly); V in fp16.
// Each warp computes S = Q K^T with ldmatrix-fed m16n8k16 MMAs, an online
// softmax in the log2 domain, and O += P V in fp16 (V fragments via
// ldmatrix.trans).  Query tiles are scheduled longest-first (causal work
// grows with the position).
#include <math.h>

#include "kvq_internal.cuh"
#include "reconstruct.cuh"

namespace kvq {
namespace {

template <int D>
struct PCfg {
  static constexpr int WARPS = D == 256 ? 4 : 8;
  static constexpr int ROWS = WARPS * 16;
  // tokens per KV tile (16 at D = 256: two CTAs fit an SM)
  static constexpr int NT = D == 256 ? 16 : 64;
  static constexpr int LDS = D + 8;                   // smem row stride (bf16), 16 B pad
  static constexpr int Q_OFF = 0;
  static constexpr int K_OFF = ROWS * LDS * 2;          // bf16 high part of K
  static constexpr int KL_OFF = K_OFF + NT * LDS * 2;   // bf16 remainder K - K_hi
  static constexpr int V_OFF = KL_OFF + NT * LDS * 2;   // fp16 V
  static constexpr int TOTAL = V_OFF + NT * LDS * 2;
  // KVarN: fp32 rows of one reconstructed tile before the inverse Hadamard
  static constexpr int SCR_OFF = TOTAL;
  // KVarN: fp32 scratch for rotating full-precision tiles, then the bf16
  // remainder of the rotated queries
  static constexpr int QL_OFF = SCR_OFF + NT * D * 4;
  static constexpr int TOTAL_KVARN = QL_OFF + ROWS * LDS * 2;
  static_assert(QL_OFF - K_OFF >= WARPS * 8 * D * 4, "half of each warp's output fits the K/V area");
  static constexpr int THREADS = WARPS * 32;
};

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void ldsm_x4(uint32_t r[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]) : "r"(smem_u32(p)));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t r[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]) : "r"(smem_u32(p)));
}
__device__ __forceinline__ void mma16816(float c[4], const uint32_t a[4], uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void mma16816_f16(float c[4], const uint32_t a[4], uint32_t b0,
                                             uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}
__device__ __forceinline__ uint32_t pack_f16(float lo, float hi) {
  __half2 v = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}
// Store 8 reconstructed values: keys as bf16 high part + bf16 remainder
// (about 16 significant bits), values as fp16.
__device__ __forceinline__ void store_k8(const float v[8], __nv_bfloat16* hi, __nv_bfloat16* lo) {
  uint32_t h[4], l[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const __nv_bfloat162 hb = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
    const float2 hf = __bfloat1622float2(hb);
    h[i] = *reinterpret_cast<const uint32_t*>(&hb);
    l[i] = pack_bf16(v[2 * i] - hf.x, v[2 * i + 1] - hf.y);
  }
  *reinterpret_cast<uint4*>(hi) = make_uint4(h[0], h[1], h[2], h[3]);
  *reinterpret_cast<uint4*>(lo) = make_uint4(l[0], l[1], l[2], l[3]);
}
__device__ __forceinline__ void store_v8(const float v[8], __half* dst) {
  *reinterpret_cast<uint4*>(dst) = make_uint4(pack_f16(v[0], v[1]), pack_f16(v[2], v[3]),
                                              pack_f16(v[4], v[5]), pack_f16(v[6], v[7]));
}

// In-warp normalised Hadamard transform of one row of D values held as
// x[i] = row[lane + 32 i]: butterflies (a + b, a - b) for h = 1 .. D/2 (lanes,
// then slots), then 1/sqrt(D).  H / sqrt(D) is symmetric and orthonormal, so
// it is its own inverse and q . k = (H q) . (H k) / D.
template <int D>
__device__ __forceinline__ void fwht_warp(float (&x)[D / 32], int lane, float inv_sqrt_d) {
  constexpr int NS = D / 32;
#pragma unroll
  for (int h = 1; h < 32; h <<= 1)
#pragma unroll
    for (int i = 0; i < NS; ++i) {
      const float y = __shfl_xor_sync(0xffffffffu, x[i], h);
      x[i] = (lane & h) ? y - x[i] : x[i] + y;
    }
#pragma unroll
  for (int hs = 1; hs < NS; hs <<= 1)
#pragma unroll
    for (int i = 0; i < NS; ++i)
      if (!(i & hs)) {
        const float a = x[i], c = x[i + hs];
        x[i] = a + c;
        x[i + hs] = a - c;
      }
#pragma unroll
  for (int i = 0; i < NS; ++i) x[i] *= inv_sqrt_d;
}

// KVarN, attended in the rotated basis: tokens [t0, t0 + NT) into dst [NT][LDS]
// bf16.  Coded tokens are stored rotated (Section 3.1: r_t c_j (s code + m)),
// so they are reconstructed as they are; sinks and staged tokens are stored
// in the original basis and are rotated forward here (fp32 butterflies in
// `scr` [NT][D]).  The queries are rotated once and the output rotated back.
template <int D, int NT, int THREADS>
__device__ void kvarn_tile(const Geom& g, int which, int b, int h, int t0, int T,
                           __nv_bfloat16* khi, __nv_bfloat16* klo, __half* vdst, int lds,
                           float* scr, float inv_sqrt_d) {
  const int G = g.G, bits = which ? g.vb : g.kb, S = g.S;
  const int nbq = kvarn_nblocks(T, S, G) * G;
  const int P_CODES = which ? KVQ_PLANE_V_CODES : KVQ_PLANE_K_CODES;
  const int P_SCALE = which ? KVQ_PLANE_V_SCALE : KVQ_PLANE_K_SCALE;
  const int P_ZERO = which ? KVQ_PLANE_V_ZERO : KVQ_PLANE_K_ZERO;
  const int P_FULL = which ? KVQ_PLANE_V_FULL : KVQ_PLANE_K_FULL;
  const int P_PEND = which ? KVQ_PLANE_V_PEND : KVQ_PLANE_K_PEND;
  const int P_ROW = which ? KVQ_PLANE_V_ROW : KVQ_PLANE_K_ROW;
  const int P_COL = which ? KVQ_PLANE_V_COL : KVQ_PLANE_K_COL;
  const unsigned mask = (1u << bits) - 1;
  // a tile with full-precision rows goes through the scratch and is rotated
  const bool all_coded = t0 >= S && t0 + NT <= S + nbq && t0 + NT <= T;
  for (int i = threadIdx.x; i < NT * (D / 8); i += THREADS) {
    const int r = i / (D / 8), c = i % (D / 8), t = t0 + r;
    float v[8];
    const bool coded = t < T && t >= S && t - S < nbq;
    if (t >= T) {
#pragma unroll
      for (int e = 0; e < 8; ++e) v[e] = 0.f;
    } else if (!coded) {
      const __nv_bfloat16* src = t < S
          ? plane_ptr<__nv_bfloat16>(g, P_FULL, b, h, t, 8 * c)
          : plane_ptr<__nv_bfloat16>(g, P_PEND, b, h, (t - S) % G, 8 * c);
      const uint4 u = *reinterpret_cast<const uint4*>(src);
      const __nv_bfloat16* e8 = reinterpret_cast<const __nv_bfloat16*>(&u);
#pragma unroll
      for (int e = 0; e < 8; ++e) v[e] = __bfloat162float(e8[e]);
    } else {
      const int qi = t - S;
      const uint8_t* row = plane_ptr<uint8_t>(g, P_CODES, b, h, qi);
      uint64_t w;
      if (bits == 4) w = *reinterpret_cast<const uint32_t*>(row + 4 * c);
      else if (bits == 2) w = *reinterpret_cast<const uint16_t*>(row + 2 * c);
      else w = *reinterpret_cast<const uint64_t*>(row + 8 * c);
      const int grp = (8 * c) / G;
      const float sc = __half2float(*plane_ptr<__half>(g, P_SCALE, b, h, qi, grp));
      const float mz = __half2float(*plane_ptr<__half>(g, P_ZERO, b, h, qi, grp));
      const float rr = __half2float(*plane_ptr<__half>(g, P_ROW, b, h, 0, qi));
      const uint4 cu = *reinterpret_cast<const uint4*>(plane_ptr<__half>(g, P_COL, b, h, qi / G, 8 * c));
      const __half* c8 = reinterpret_cast<const __half*>(&cu);
#pragma unroll
      for (int e = 0; e < 8; ++e)
        v[e] = rr * __half2float(c8[e]) * ((float)((w >> (e * bits)) & mask) * sc + mz);
    }
    if (all_coded) {
      if (which == 0) store_k8(v, khi + r * lds + 8 * c, klo + r * lds + 8 * c);
      else store_v8(v, vdst + r * lds + 8 * c);
    } else {
      float* sr = scr + r * D + 8 * c;
#pragma unroll
      for (int e = 0; e < 8; ++e) sr[e] = v[e];
    }
  }
  if (all_coded) return;
  __syncthreads();
  // forward rotation of the full-precision rows (butterflies h = 1 .. D/2)
  for (int hs = 1; hs < D; hs <<= 1) {
    for (int p = threadIdx.x; p < NT * D / 2; p += THREADS) {
      const int r = p / (D / 2), k = p % (D / 2), t = t0 + r;
      if (t >= T || (t >= S && t - S < nbq)) continue;
      const int j = (k / hs) * 2 * hs + (k % hs);
      const float a = scr[r * D + j], c = scr[r * D + j + hs];
      scr[r * D + j] = a + c;
      scr[r * D + j + hs] = a - c;
    }
    __syncthreads();
  }
  for (int i = threadIdx.x; i < NT * (D / 8); i += THREADS) {
    const int r = i / (D / 8), c = i % (D / 8), t = t0 + r;
    const float f = (t < T && !(t >= S && t - S < nbq)) ? inv_sqrt_d : 1.f;
    const float* sr = scr + r * D + 8 * c;
    float v[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) v[e] = sr[e] * f;
    if (which == 0) store_k8(v, khi + r * lds + 8 * c, klo + r * lds + 8 * c);
    else store_v8(v, vdst + r * lds + 8 * c);
  }
}

// KVarN tile with full-precision rows (sinks, staged tokens) among its NT
// tokens: a warp per token builds the key and value rows in the layout
// x[i] = row[lane + 32 i]; coded tokens are reconstructed as stored (rotated),
// full-precision ones are rotated forward in registers by fwht_warp (the same
// butterflies, in the same order, as the rotation of the queries), so the tile
// needs no scratch and no CTA barrier.
template <int D, int NT, int THREADS>
__device__ __noinline__ void kvarn_tile_rows(const Geom& g, int b, int h, int t0, int T,
                                __nv_bfloat16* khi, __nv_bfloat16* klo, __half* vdst, int lds,
                                float inv_sqrt_d) {
  constexpr int NS = D / 32, NW = THREADS / 32;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = g.G, S = g.S;
  const int nbq = kvarn_nblocks(T, S, G) * G;
  for (int r = warp; r < NT; r += NW) {
    const int t = t0 + r;
    float kx[NS], vx[NS];
    if (t >= T) {
#pragma unroll
      for (int i = 0; i < NS; ++i) kx[i] = vx[i] = 0.f;
    } else if (t < S || t - S >= nbq) {
      const __nv_bfloat16* ks = t < S ? plane_ptr<__nv_bfloat16>(g, KVQ_PLANE_K_FULL, b, h, t, 0)
                                      : plane_ptr<__nv_bfloat16>(g, KVQ_PLANE_K_PEND, b, h, (t - S) % G, 0);
      const __nv_bfloat16* vs = t < S ? plane_ptr<__nv_bfloat16>(g, KVQ_PLANE_V_FULL, b, h, t, 0)
                                      : plane_ptr<__nv_bfloat16>(g, KVQ_PLANE_V_PEND, b, h, (t - S) % G, 0);
#pragma unroll
      for (int i = 0; i < NS; ++i) {
        kx[i] = __bfloat162float(ks[lane + 32 * i]);
        vx[i] = __bfloat162float(vs[lane + 32 * i]);
      }
      fwht_warp<D>(kx, lane, inv_sqrt_d);
      fwht_warp<D>(vx, lane, inv_sqrt_d);
    } else {
      const int qi = t - S;
#pragma unroll
      for (int which = 0; which < 2; ++which) {
        const int bits = which ? g.vb : g.kb;
        const unsigned mask = (1u << bits) - 1;
        const uint8_t* row = plane_ptr<uint8_t>(g, which ? KVQ_PLANE_V_CODES : KVQ_PLANE_K_CODES, b, h, qi);
        const float rr = __half2float(*plane_ptr<__half>(g, which ? KVQ_PLANE_V_ROW : KVQ_PLANE_K_ROW, b, h, 0, qi));
        const __half* col = plane_ptr<__half>(g, which ? KVQ_PLANE_V_COL : KVQ_PLANE_K_COL, b, h, qi / G, 0);
        const __half* scp = plane_ptr<__half>(g, which ? KVQ_PLANE_V_SCALE : KVQ_PLANE_K_SCALE, b, h, qi, 0);
        const __half* zp = plane_ptr<__half>(g, which ? KVQ_PLANE_V_ZERO : KVQ_PLANE_K_ZERO, b, h, qi, 0);
#pragma unroll
        for (int i = 0; i < NS; ++i) {
          const int j = lane + 32 * i, bit = j * bits;
          const unsigned code = ((unsigned)row[bit >> 3] >> (bit & 7)) & mask;
          const float sc = __half2float(scp[j / G]), mz = __half2float(zp[j / G]);
          const float v = rr * __half2float(col[j]) * ((float)code * sc + mz);
          if (which) vx[i] = v;
          else kx[i] = v;
        }
      }
    }
#pragma unroll
    for (int i = 0; i < NS; ++i) {
      const int j = lane + 32 * i;
      const __nv_bfloat16 hb = __float2bfloat16_rn(kx[i]);
      khi[r * lds + j] = hb;
      klo[r * lds + j] = __float2bfloat16_rn(kx[i] - __bfloat162float(hb));
      vdst[r * lds + j] = __float2half_rn(vx[i]);
    }
  }
}

// KVarN tile whose tokens are all coded (stored rotated: r_t c_j (s code + m)),
// keys and values in one pass.  A thread keeps one 8-channel chunk for all
// of its tokens; the tile lies inside one column-scale block (NT divides the
// block length G and the sinks end on a tile boundary), so the chunk's
// column scales are loaded once.
template <int D, int NT, int THREADS>
__device__ __forceinline__ void kvarn_tile_coded(const Geom& g, int b, int h, int t0,
                                                 __nv_bfloat16* khi, __nv_bfloat16* klo,
                                                 __half* vdst, int lds) {
  constexpr int CH = D / 8;
  constexpr int RSTEP = THREADS / CH;
  static_assert(THREADS % CH == 0 && NT % RSTEP == 0, "whole tokens per pass");
  const int c = threadIdx.x % CH, r0 = threadIdx.x / CH;
  const int kb = g.kb, vb = g.vb, grp = (8 * c) / g.G;
  const unsigned kmask = (1u << kb) - 1, vmask = (1u << vb) - 1;
  const int blk = (t0 - g.S) / g.G;
  const uint4 kcu = *reinterpret_cast<const uint4*>(plane_ptr<__half>(g, KVQ_PLANE_K_COL, b, h, blk, 8 * c));
  const uint4 vcu = *reinterpret_cast<const uint4*>(plane_ptr<__half>(g, KVQ_PLANE_V_COL, b, h, blk, 8 * c));
#pragma unroll 1
  for (int k = 0; k < NT / RSTEP; ++k) {
    const int r = r0 + k * RSTEP, qi = t0 + r - g.S;
    const uint8_t* krow = plane_ptr<uint8_t>(g, KVQ_PLANE_K_CODES, b, h, qi);
    const uint8_t* vrow = plane_ptr<uint8_t>(g, KVQ_PLANE_V_CODES, b, h, qi);
    const uint32_t kw = kb == 4 ? *reinterpret_cast<const uint32_t*>(krow + 4 * c)
                                : *reinterpret_cast<const uint16_t*>(krow + 2 * c);
    const uint32_t vw = vb == 4 ? *reinterpret_cast<const uint32_t*>(vrow + 4 * c)
                                : *reinterpret_cast<const uint16_t*>(vrow + 2 * c);
    const float ks = __half2float(*plane_ptr<__half>(g, KVQ_PLANE_K_SCALE, b, h, qi, grp));
    const float kz = __half2float(*plane_ptr<__half>(g, KVQ_PLANE_K_ZERO, b, h, qi, grp));
    const float vs = __half2float(*plane_ptr<__half>(g, KVQ_PLANE_V_SCALE, b, h, qi, grp));
    const float vz = __half2float(*plane_ptr<__half>(g, KVQ_PLANE_V_ZERO, b, h, qi, grp));
    const float kr = __half2float(*plane_ptr<__half>(g, KVQ_PLANE_K_ROW, b, h, 0, qi));
    const float vr = __half2float(*plane_ptr<__half>(g, KVQ_PLANE_V_ROW, b, h, 0, qi));
    const __half2* kc2 = reinterpret_cast<const __half2*>(&kcu);
    const __half2* vc2 = reinterpret_cast<const __half2*>(&vcu);
    float kv[8], vv[8];
#pragma unroll
    for (int e2 = 0; e2 < 4; ++e2) {
      const float2 kc = __half22float2(kc2[e2]), vc = __half22float2(vc2[e2]);
      kv[2 * e2] = kr * kc.x * ((float)((kw >> (2 * e2 * kb)) & kmask) * ks + kz);
      kv[2 * e2 + 1] = kr * kc.y * ((float)((kw >> ((2 * e2 + 1) * kb)) & kmask) * ks + kz);
      vv[2 * e2] = vr * vc.x * ((float)((vw >> (2 * e2 * vb)) & vmask) * vs + vz);
      vv[2 * e2 + 1] = vr * vc.y * ((float)((vw >> ((2 * e2 + 1) * vb)) & vmask) * vs + vz);
    }
    store_k8(kv, khi + r * lds + 8 * c, klo + r * lds + 8 * c);
    store_v8(vv, vdst + r * lds + 8 * c);
  }
}

// KIVI with BITS-bit keys and values: tokens [t0, t0 + NT) into the K high /
// remainder and V tiles.  A thread keeps one 8-channel chunk for all of its
// tokens, so the keys' per-channel block scales and offsets (one row per 32
// tokens) are loaded once per block, and the plane rows are addressed from
// per-head bases.  Tokens from tq on are the full-precision residual ring.
template <int D, int BITS, int NT, int THREADS>
__device__ __forceinline__ void kivi_tile(const Geom& g, int b, int h, int t0, int T, int tq,
                                          __nv_bfloat16* khi, __nv_bfloat16* klo, __half* vdst,
                                          int lds) {
  constexpr int CH = D / 8;
  constexpr int RSTEP = THREADS / CH;                 // token step between a thread's items
  static_assert(THREADS % CH == 0 && NT % RSTEP == 0, "whole tokens per pass");
  constexpr unsigned mask = (1u << BITS) - 1;
  const int c = threadIdx.x % CH, r0 = threadIdx.x / CH;
  int cur_blk = -1;
  uint4 su = make_uint4(0, 0, 0, 0), zu = make_uint4(0, 0, 0, 0);   // block scales, offsets (fp16)
#pragma unroll 1
  for (int k = 0; k < NT / RSTEP; ++k) {
    const int r = r0 + k * RSTEP, t = t0 + r;
    float kv[8], vv[8];
    if (t >= T) {
#pragma unroll
      for (int e = 0; e < 8; ++e) kv[e] = vv[e] = 0.f;
    } else if (t >= tq) {
      const int slot = t % g.ring;
      const uint4 ku = *reinterpret_cast<const uint4*>(plane_ptr<__nv_bfloat16>(g, KVQ_PLANE_K_FULL, b, h, slot, 8 * c));
      const uint4 vu = *reinterpret_cast<const uint4*>(plane_ptr<__nv_bfloat16>(g, KVQ_PLANE_V_FULL, b, h, slot, 8 * c));
      const __nv_bfloat16* k8 = reinterpret_cast<const __nv_bfloat16*>(&ku);
      const __nv_bfloat16* v8 = reinterpret_cast<const __nv_bfloat16*>(&vu);
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        kv[e] = __bfloat162float(k8[e]);
        vv[e] = __bfloat162float(v8[e]);
      }
    } else {
      const int blk = t / 32;
      if (blk != cur_blk) {                           // the keys' block scales of these channels
        cur_blk = blk;
        su = *reinterpret_cast<const uint4*>(plane_ptr<__half>(g, KVQ_PLANE_K_SCALE, b, h, blk, 8 * c));
        zu = *reinterpret_cast<const uint4*>(plane_ptr<__half>(g, KVQ_PLANE_K_ZERO, b, h, blk, 8 * c));
      }
      const uint8_t* kr = plane_ptr<uint8_t>(g, KVQ_PLANE_K_CODES, b, h, t) + (BITS == 4 ? 4 : 2) * c;
      const uint8_t* vr = plane_ptr<uint8_t>(g, KVQ_PLANE_V_CODES, b, h, t) + (BITS == 4 ? 4 : 2) * c;
      const uint32_t kw = BITS == 4 ? *reinterpret_cast<const uint32_t*>(kr)
                                    : *reinterpret_cast<const uint16_t*>(kr);
      const uint32_t vw = BITS == 4 ? *reinterpret_cast<const uint32_t*>(vr)
                                    : *reinterpret_cast<const uint16_t*>(vr);
      const float vs = __half2float(*plane_ptr<__half>(g, KVQ_PLANE_V_SCALE, b, h, t, c / 4));
      const float vz = __half2float(*plane_ptr<__half>(g, KVQ_PLANE_V_ZERO, b, h, t, c / 4));
      const __half2* s2 = reinterpret_cast<const __half2*>(&su);
      const __half2* z2 = reinterpret_cast<const __half2*>(&zu);
#pragma unroll
      for (int e2 = 0; e2 < 4; ++e2) {
        const float2 sf = __half22float2(s2[e2]), zf = __half22float2(z2[e2]);
        kv[2 * e2] = (float)((kw >> (2 * e2 * BITS)) & mask) * sf.x + zf.x;
        kv[2 * e2 + 1] = (float)((kw >> ((2 * e2 + 1) * BITS)) & mask) * sf.y + zf.y;
        vv[2 * e2] = (float)((vw >> (2 * e2 * BITS)) & mask) * vs + vz;
        vv[2 * e2 + 1] = (float)((vw >> ((2 * e2 + 1) * BITS)) & mask) * vs + vz;
      }
    }
    store_k8(kv, khi + r * lds + 8 * c, klo + r * lds + 8 * c);
    store_v8(vv, vdst + r * lds + 8 * c);
  }
}

// KIVIB: 0 = any format (tiles through deq8 or kvarn_tile); 2 or 4 = a KIVI
// cache with KIVIB-bit keys and values (tiles through kivi_tile).
template <int D, int KIVIB>
__global__ void __launch_bounds__(PCfg<D>::THREADS, D >= 128 ? 2 : 1)
attend_prefill_mma_kernel(Geom g, const __nv_bfloat16* __restrict__ q, int L, float scale,
                          __nv_bfloat16* __restrict__ out, int nq, float inv_sqrt_d) {
  pdl_wait();
  pdl_trigger();
  using C = PCfg<D>;
  constexpr int NT = C::NT, LDS = C::LDS, NTN = NT / 8;   // n-tiles of 8 tokens
  extern __shared__ __align__(16) unsigned char smem[];
  __nv_bfloat16* Qs = reinterpret_cast<__nv_bfloat16*>(smem + C::Q_OFF);
  __nv_bfloat16* Ks = reinterpret_cast<__nv_bfloat16*>(smem + C::K_OFF);
  __nv_bfloat16* Kl = reinterpret_cast<__nv_bfloat16*>(smem + C::KL_OFF);
  __half* Vs = reinterpret_cast<__half*>(smem + C::V_OFF);

  const int nqt = gridDim.x;
  const int qtile = nqt - 1 - blockIdx.x;             // longest first
  const int hkv = blockIdx.y, b = blockIdx.z;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gid = lane >> 2, tid = lane & 3;
  const int grp = g.Hq / g.H;
  const int T = cache_tokens(g);
  const int tq = g.fmt == KVQ_FMT_KIVI ? kivi_tq(T, g.R, g.G) : T;
  const int q0 = qtile * nq;
  const int nql = min(nq, L - q0);
  const int pos_first = T - L + q0;
  const int t_end = pos_first + nql;                  // keys [0, t_end)

  // queries -> shared memory (zero rows beyond the heads or queries)
  for (int i = threadIdx.x; i < C::ROWS * (D / 8); i += C::THREADS) {
    const int r = i / (D / 8), c = i % (D / 8);
    const int hl = r / nq, qi = r % nq;
    uint4 v = make_uint4(0, 0, 0, 0);
    if (hl < grp && qi < nql)
      v = *reinterpret_cast<const uint4*>(
          q + (((int64_t)b * g.Hq + hkv * grp + hl) * L + q0 + qi) * D + 8 * c);
    *reinterpret_cast<uint4*>(Qs + r * LDS + 8 * c) = v;
  }
  const bool kvarn = KIVIB == 0 && g.fmt == KVQ_FMT_KVARN;
  __nv_bfloat16* Ql = reinterpret_cast<__nv_bfloat16*>(smem + C::QL_OFF);
  if (kvarn) {
    // rotate the query rows: high part in Qs, bf16 remainder in Ql
    __syncthreads();
    for (int r = warp; r < C::ROWS; r += C::WARPS) {
      float x[D / 32];
#pragma unroll
      for (int i = 0; i < D / 32; ++i) x[i] = __bfloat162float(Qs[r * LDS + lane + 32 * i]);
      fwht_warp<D>(x, lane, inv_sqrt_d);
#pragma unroll
      for (int i = 0; i < D / 32; ++i) {
        const __nv_bfloat16 hb = __float2bfloat16_rn(x[i]);
        Qs[r * LDS + lane + 32 * i] = hb;
        Ql[r * LDS + lane + 32 * i] = __float2bfloat16_rn(x[i] - __bfloat162float(hb));
      }
    }
  }
  // this thread's two rows: positions (or -1 for padding rows)
  int pos[2];
  for (int rr = 0; rr < 2; ++rr) {
    const int r = warp * 16 + gid + 8 * rr;
    const int hl = r / nq, qi = r % nq;
    pos[rr] = (hl < grp && qi < nql) ? pos_first + qi : -1;
  }
  const int warp_pos_max = [&] {
    int m = -1;
    for (int i = 0; i < 16; ++i) {
      const int r = warp * 16 + i;
      const int hl = r / nq, qi = r % nq;
      if (hl < grp && qi < nql) m = max(m, pos_first + qi);
    }
    return m;
  }();
  const float c2 = scale * 1.4426950408889634f;
  float m_run[2] = {-INFINITY, -INFINITY}, l_run[2] = {0.f, 0.f};
  float o[D / 8][4];
#pragma unroll
  for (int j = 0; j < D / 8; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;

  for (int t0 = 0; t0 < t_end; t0 += NT) {
    __syncthreads();                                  // previous tile consumed
    if (KIVIB != 0) {
      kivi_tile<D, KIVIB == 0 ? 2 : KIVIB, NT, C::THREADS>(g, b, hkv, t0, T, tq, Ks, Kl, Vs, LDS);
    } else if (D != 128 && g.fmt == KVQ_FMT_KVARN && t0 >= g.S && t0 + NT <= T &&
               t0 + NT <= g.S + kvarn_nblocks(T, g.S, g.G) * g.G && g.G % NT == 0 && g.S % NT == 0) {
      kvarn_tile_coded<D, NT, C::THREADS>(g, b, hkv, t0, Ks, Kl, Vs, LDS);
    } else if (g.fmt == KVQ_FMT_KVARN && D != 128) {
      kvarn_tile_rows<D, NT, C::THREADS>(g, b, hkv, t0, T, Ks, Kl, Vs, LDS, inv_sqrt_d);
    } else if (g.fmt == KVQ_FMT_KVARN) {
      float* scr = reinterpret_cast<float*>(smem + C::SCR_OFF);
      kvarn_tile<D, NT, C::THREADS>(g, 0, b, hkv, t0, T, Ks, Kl, Vs, LDS, scr, inv_sqrt_d);
      __syncthreads();
      kvarn_tile<D, NT, C::THREADS>(g, 1, b, hkv, t0, T, Ks, Kl, Vs, LDS, scr, inv_sqrt_d);
    } else {
      for (int i = threadIdx.x; i < NT * (D / 8); i += C::THREADS) {
        const int r = i / (D / 8), c = i % (D / 8);
        float v[8];
        deq8(g, 0, b, hkv, t0 + r, c, T, tq, v);
        store_k8(v, Ks + r * LDS + 8 * c, Kl + r * LDS + 8 * c);
        deq8(g, 1, b, hkv, t0 + r, c, T, tq, v);
        store_v8(v, Vs + r * LDS + 8 * c);
      }
    }
    __syncthreads();
    if (warp_pos_max < t0) continue;                  // tile entirely in this warp's future
    // ---- S = Q K^T ----
    float s[NTN][4];
#pragma unroll
    for (int j = 0; j < NTN; ++j) s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.f;
#pragma unroll
    for (int ks = 0; ks < D / 16; ++ks) {
      uint32_t a[4], al[4];
      const int qoff = (warp * 16 + (lane & 15)) * LDS + 16 * ks + (lane >> 4) * 8;
      ldsm_x4(a, Qs + qoff);
      if (kvarn) ldsm_x4(al, Ql + qoff);
#pragma unroll
      for (int np = 0; np < NTN / 2; ++np) {
        uint32_t bq[4], bl[4];
        const int j = lane >> 3, i = lane & 7;
        const int off = ((2 * np + (j >> 1)) * 8 + i) * LDS + 16 * ks + (j & 1) * 8;
        ldsm_x4(bq, Ks + off);
        ldsm_x4(bl, Kl + off);
        mma16816(s[2 * np], a, bq[0], bq[1]);
        mma16816(s[2 * np + 1], a, bq[2], bq[3]);
        mma16816(s[2 * np], a, bl[0], bl[1]);
        mma16816(s[2 * np + 1], a, bl[2], bl[3]);
        if (kvarn) {
          mma16816(s[2 * np], al, bq[0], bq[1]);
          mma16816(s[2 * np + 1], al, bq[2], bq[3]);
        }
      }
    }
    // ---- mask, online softmax ----
    const bool diag = t0 + NT - 1 > pos_first;         // some key may be in a row's future
    float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
    for (int j = 0; j < NTN; ++j)
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int rr = i >> 1;
        const int t = t0 + 8 * j + 2 * tid + (i & 1);
        float v = s[j][i] * c2;
        if (diag && t > pos[rr]) v = -INFINITY;
        s[j][i] = v;
        mx[rr] = fmaxf(mx[rr], v);
      }
    float alpha[2];
#pragma unroll
    for (int rr = 0; rr < 2; ++rr) {
      mx[rr] = fmaxf(mx[rr], __shfl_xor_sync(0xffffffffu, mx[rr], 1));
      mx[rr] = fmaxf(mx[rr], __shfl_xor_sync(0xffffffffu, mx[rr], 2));
      const float mn = fmaxf(m_run[rr], mx[rr]);
      alpha[rr] = mn == -INFINITY ? 1.f : exp2f(m_run[rr] - mn);
      m_run[rr] = mn;
      l_run[rr] *= alpha[rr];
    }
#pragma unroll
    for (int j = 0; j < D / 8; ++j) {
      o[j][0] *= alpha[0]; o[j][1] *= alpha[0];
      o[j][2] *= alpha[1]; o[j][3] *= alpha[1];
    }
    uint32_t pa[NT / 16][4];
#pragma unroll
    for (int j = 0; j < NTN; ++j) {
      float p[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float mr = m_run[i >> 1];
        p[i] = s[j][i] == -INFINITY ? 0.f : exp2f(s[j][i] - mr);
        l_run[i >> 1] += p[i];
      }
      // A fragment of k-step j/2: n-tile 2k -> a0 (row gid), a1 (row gid+8);
      // n-tile 2k+1 -> a2, a3
      pa[j >> 1][(j & 1) * 2 + 0] = pack_f16(p[0], p[1]);
      pa[j >> 1][(j & 1) * 2 + 1] = pack_f16(p[2], p[3]);
    }
    // ---- O += P V ----
#pragma unroll
    for (int kt = 0; kt < NT / 16; ++kt) {
#pragma unroll
      for (int nd = 0; nd < D / 8; nd += 2) {
        uint32_t bv[4];
        const int j = lane >> 3, i = lane & 7;
        ldsm_x4_t(bv, Vs + (16 * kt + (j & 1) * 8 + i) * LDS + 8 * (nd + (j >> 1)));
        mma16816_f16(o[nd], pa[kt], bv[0], bv[1]);
        mma16816_f16(o[nd + 1], pa[kt], bv[2], bv[3]);
      }
    }
  }
  // ---- normalise and store ----
#pragma unroll
  for (int rr = 0; rr < 2; ++rr) {
    l_run[rr] += __shfl_xor_sync(0xffffffffu, l_run[rr], 1);
    l_run[rr] += __shfl_xor_sync(0xffffffffu, l_run[rr], 2);
  }
  if (kvarn) {
    // normalised rotated rows -> fp32 shared memory (each warp its own 8
    // rows of the K/V area at a time), then the warp rotates them back
    float* os = reinterpret_cast<float*>(smem + C::K_OFF) + warp * 8 * D;   // [8][D]
    __syncthreads();                                  // every warp is done with K and V
#pragma unroll
    for (int rr = 0; rr < 2; ++rr) {
      const float inv = l_run[rr] > 0.f ? 1.f / l_run[rr] : 0.f;
#pragma unroll
      for (int j = 0; j < D / 8; ++j) {
        os[gid * D + 8 * j + 2 * tid] = o[j][2 * rr] * inv;
        os[gid * D + 8 * j + 2 * tid + 1] = o[j][2 * rr + 1] * inv;
      }
      __syncwarp();
      for (int k = 0; k < 8; ++k) {
        const int r = warp * 16 + 8 * rr + k;
        const int hl = r / nq, qi = r % nq;
        if (hl >= grp || qi >= nql) continue;
        float x[D / 32];
#pragma unroll
        for (int i = 0; i < D / 32; ++i) x[i] = os[k * D + lane + 32 * i];
        fwht_warp<D>(x, lane, inv_sqrt_d);
        __nv_bfloat16* orow = out + (((int64_t)b * g.Hq + hkv * grp + hl) * L + q0 + qi) * D;
#pragma unroll
        for (int i = 0; i < D / 32; ++i) orow[lane + 32 * i] = __float2bfloat16_rn(x[i]);
      }
      __syncwarp();                                   // the rows are read before the next half
    }
    return;
  }
#pragma unroll
  for (int rr = 0; rr < 2; ++rr) {
    const int r = warp * 16 + gid + 8 * rr;
    const int hl = r / nq, qi = r % nq;
    if (hl >= grp || qi >= nql) continue;
    const float inv = 1.f / l_run[rr];
    __nv_bfloat16* orow = out + (((int64_t)b * g.Hq + hkv * grp + hl) * L + q0 + qi) * D;
#pragma unroll
    for (int j = 0; j < D / 8; ++j)
      *reinterpret_cast<uint32_t*>(orow + 8 * j + 2 * tid) =
          pack_bf16(o[j][2 * rr] * inv, o[j][2 * rr + 1] * inv);
  }
}

template <int D>
cudaError_t launch_d(const Geom& g, const void* q, int L, float scale, void* out,
                     cudaStream_t s) {
  using C = PCfg<D>;
  const int grp = g.Hq / g.H;
  const int nq = C::ROWS / grp;
  auto kern = g.fmt == KVQ_FMT_KIVI && g.kb == g.vb && g.kb == 2 ? attend_prefill_mma_kernel<D, 2>
            : g.fmt == KVQ_FMT_KIVI && g.kb == g.vb && g.kb == 4 ? attend_prefill_mma_kernel<D, 4>
                                                                 : attend_prefill_mma_kernel<D, 0>;
  const int smem = g.fmt == KVQ_FMT_KVARN ? C::TOTAL_KVARN : C::TOTAL;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  const float inv_sqrt_d = (float)(1.0 / sqrt((double)D));
  dim3 grid((L + nq - 1) / nq, g.H, g.B);
  launch_pdl(kern, dim3(grid), dim3(C::THREADS), (size_t)smem, s, g,
             reinterpret_cast<const __nv_bfloat16*>(q), L, scale,
             reinterpret_cast<__nv_bfloat16*>(out), nq, inv_sqrt_d);
  return cudaGetLastError();
}

}  // namespace

bool prefill_mma_supported(const Geom& g) {
  const bool fmt_ok = g.fmt == KVQ_FMT_AFFINE || g.fmt == KVQ_FMT_SYMMETRIC ||
                      g.fmt == KVQ_FMT_KIVI || g.fmt == KVQ_FMT_FLOAT || g.fmt == KVQ_FMT_KVARN;
  const int grp = g.Hq / g.H;
  const int rows = g.D == 256 ? 64 : 128;
  return fmt_ok && g.layout == KVQ_LAYOUT_UNIFORM && g.act == KVQ_BF16 && grp <= rows &&
         (g.D == 64 || g.D == 128 || g.D == 256);
}

cudaError_t launch_prefill_mma(const Geom& g, const void* q, int L, float scale, void* out,
                               cudaStream_t s) {
  if (g.D == 64) return launch_d<64>(g, q, L, scale, out, s);
  if (g.D == 128) return launch_d<128>(g, q, L, scale, out, s);
  return launch_d<256>(g, q, L, scale, out, s);
}

}  // namespace kvq
