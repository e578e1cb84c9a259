// Quantize-and-pack of new keys/values into the physical incremental cache
// (Section 3.1).  Every value that decides a code is computed in IEEE fp32
// with explicitly rounded operations (no contraction), in the order the cache
// format fixes, so codes and fp16 metadata are reproducible bit for bit.
#include <math.h>

#include "kvq_internal.cuh"
#include "quant_common.cuh"

namespace kvq {
namespace {
using namespace quant;

// Where token t of a (b, h) row comes from: the new input for t >= T0,
// otherwise a full-precision ring plane (KIVI residual or KVarN staging).
struct TokSrc {
  const void* x;      // [B][H][L][D] new tokens
  int T0, L;
  int ring_plane;     // plane index of the ring, -1 if none
  int ring_off, ring_rows;
};

__device__ __forceinline__ int64_t tok_elem(const Geom& g, const TokSrc& s, int b, int h,
                                            int t, const void** base) {
  if (t >= s.T0) {
    *base = s.x;
    return (((int64_t)b * g.H + h) * s.L + (t - s.T0)) * g.D;
  }
  const Plane& pl = g.pl[s.ring_plane];
  *base = pl.p;
  int slot = (t - s.ring_off) % s.ring_rows;
  return plane_index(pl, b, h, g.H, slot, 0);
}

// Load 8 consecutive activation elements (16-byte aligned) as fp32.
__device__ __forceinline__ void load8(const void* base, int64_t e, int act, float v[8]) {
  if (act == KVQ_BF16) {
    uint4 u = *reinterpret_cast<const uint4*>(reinterpret_cast<const __nv_bfloat16*>(base) + e);
    const __nv_bfloat162* p = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      float2 f = __bfloat1622float2(p[i]);
      v[2 * i] = f.x;
      v[2 * i + 1] = f.y;
    }
  } else {
    const float4* p = reinterpret_cast<const float4*>(reinterpret_cast<const float*>(base) + e);
    float4 a = p[0], b = p[1];
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
  }
}

// ---------------------------------------------------------------------------
// Per-token grouped coding: AFFINE / SYMMETRIC keys and values, KIVI values.
// A group of G elements is held by G/8 consecutive lanes, 8 elements each;
// min/max (or absmax) is a butterfly over those lanes; each lane packs its 8
// codes LSB-first into one 16/32/64-bit store.  blockIdx.y selects keys (0)
// or values (1).  kivi = 1: code the values of the KIVI blocks that this
// append completes (tokens [q0, q1), read from the residual ring or the
// input); else code the new tokens [T0, T0 + L).  A grid-stride loop over
// 8-element chunks with 32-bit indices (the host bounds the chunk count).
// ---------------------------------------------------------------------------
// Code tokens [t_begin, t_begin + ntok) of the (b, h) row of keys (which = 0)
// or values; src.T0 is the row's first new token.  Stores go through
// tok_ptr, so the same code serves every token layout.
__device__ __forceinline__ void pack_rows(const Geom& g, const TokSrc& src, int b, int h,
                                          int t_begin, int ntok, int which, int sym, int lcpt,
                                          int llpg) {
  const int bits = which ? g.vb : g.kb;
  const int lane = threadIdx.x & 31;
  const int cpt = 1 << lcpt;               // 8-element chunks per token (D / 8)
  const int total = ntok << lcpt;          // chunks of this (b, h) row
  const int codes_plane = which ? KVQ_PLANE_V_CODES : KVQ_PLANE_K_CODES;
  const int scale_plane = which ? KVQ_PLANE_V_SCALE : KVQ_PLANE_K_SCALE;
  const int zero_plane = which ? KVQ_PLANE_V_ZERO : KVQ_PLANE_K_ZERO;
  const int stride = gridDim.x * blockDim.x;
  // chunk i = token * cpt + c8 of the row.  A warp covers 32 consecutive
  // chunks, so a group's G/8 lanes are consecutive and aligned
  for (int i0 = blockIdx.x * blockDim.x + (threadIdx.x & ~31); i0 < total; i0 += stride) {
    const int i = i0 + lane;
    const bool live = i < total;
    const int ii = live ? i : total - 1;
    const int t = t_begin + (ii >> lcpt), c8 = ii & (cpt - 1);
    const int grp = c8 >> llpg, li = c8 & ((1 << llpg) - 1);
    const void* sb;
    const int64_t e = tok_elem(g, src, b, h, t, &sb) + c8 * 8;
    float v[8];
    load8(sb, e, g.act, v);
    float lo = v[0], hi = sym ? fabsf(v[0]) : v[0];
#pragma unroll
    for (int i = 1; i < 8; ++i) {
      if (sym) hi = fmaxf(hi, fabsf(v[i]));
      else { lo = fminf(lo, v[i]); hi = fmaxf(hi, v[i]); }
    }
    for (int off = (1 << llpg) >> 1; off > 0; off >>= 1) {
      lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, off));
      hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, off));
    }
    float s;
    uint64_t word;
    if (sym) {
      word = bits == 2 ? code8<2, true>(v, lo, hi, &s)
           : bits == 4 ? code8<4, true>(v, lo, hi, &s) : code8<8, true>(v, lo, hi, &s);
    } else {
      word = bits == 2 ? code8<2, false>(v, lo, hi, &s)
           : bits == 4 ? code8<4, false>(v, lo, hi, &s) : code8<8, false>(v, lo, hi, &s);
    }
    if (!live) continue;
    uint8_t* crow = tok_ptr<uint8_t>(g, codes_plane, b, h, t);
    const int byte0 = c8 * bits;
    if (bits == 2) *reinterpret_cast<uint16_t*>(crow + byte0) = (uint16_t)word;
    else if (bits == 4) *reinterpret_cast<uint32_t*>(crow + byte0) = (uint32_t)word;
    else *reinterpret_cast<uint64_t*>(crow + byte0) = word;
    if (li == 0) {
      *tok_ptr<__half>(g, scale_plane, b, h, t, grp) = __float2half_rn(s);
      if (!sym) *tok_ptr<__half>(g, zero_plane, b, h, t, grp) = __float2half_rn(lo + 0.0f);
    }
  }
}

// A ragged cache (layouts RAGGED and PAGED) appends per sequence: sequence b
// codes its first seq_new[b] of the L new tokens at its own positions
// seq_len[b] ..; the host has checked capacity and assigned the pages, and
// the counts advance after the append's kernels.
__global__ void pack_pertoken_kernel(Geom g, int L, TokSrc sk, TokSrc sv, int sym, int kivi,
                                     int final_kernel, int lcpt, int llpg) {
  pdl_wait();
  pdl_trigger();
  bool ok = true;
  const bool rag = g.layout != KVQ_LAYOUT_UNIFORM;
  const int T0u = rag ? 0 : append_begin(g, L, &ok);
  const int which = kivi ? 1 : blockIdx.z;
  const int b = blockIdx.y / g.H, h = blockIdx.y - b * g.H;
  int T0, n;
  append_span(g, b, L, T0u, &T0, &n);
  int t_begin = T0, t_end = T0 + n;
  if (kivi) {
    t_begin = kivi_tq(T0, g.R, g.G);
    t_end = kivi_tq(T0 + n, g.R, g.G);
  }
  if (ok && t_end > t_begin) {
    TokSrc src = which ? sv : sk;
    src.T0 = T0;
    pack_rows(g, src, b, h, t_begin, t_end - t_begin, which, sym, lcpt, llpg);
  }
  if (final_kernel && !rag) append_arrive_spread(g.state, T0u, L, ok);
}

// Ragged appends: this append's counts (first), and the sequences' counts
// advanced by them (last).
struct SeqCounts {
  int32_t n[KVQ_MAX_SEQS];
};

__global__ void seq_counts_kernel(Geom g, SeqCounts n) {
  pdl_wait();
  pdl_trigger();
  for (int b = threadIdx.x; b < g.B; b += blockDim.x) g.seq_new[b] = n.n[b];
}

__global__ void seq_advance_kernel(Geom g) {
  pdl_wait();
  pdl_trigger();
  for (int b = threadIdx.x; b < g.B; b += blockDim.x) g.seq_len[b] += g.seq_new[b];
}

// KIVI's full-precision ring for a ragged cache: sequence b's new tokens that
// stay outside its coded prefix, token t in slot t mod (R + G).
__global__ void store_ring_ragged_kernel(Geom g, int L, const void* k, const void* v) {
  pdl_wait();
  pdl_trigger();
  const int which = blockIdx.y;
  const void* x = which ? v : k;
  const int vec_per_tok = g.D * 2 / 16;                 // bf16
  const int total = g.B * g.H * L * vec_per_tok;        // below 2^31 (checked by the host)
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < total; i += gridDim.x * blockDim.x) {
    const int vi = i % vec_per_tok;
    const int rest = i / vec_per_tok;
    const int j = rest % L, row = rest / L;
    const int h = row % g.H, b = row / g.H;
    int T0, n;
    append_span(g, b, L, 0, &T0, &n);
    const int t = T0 + j;
    if (j >= n || t < kivi_tq(T0 + n, g.R, g.G)) continue;
    const int plane = which ? KVQ_PLANE_V_FULL : KVQ_PLANE_K_FULL;
    const uint4* src = reinterpret_cast<const uint4*>(x) + ((int64_t)row * L + j) * vec_per_tok;
    uint4* dst = reinterpret_cast<uint4*>(plane_ptr<__nv_bfloat16>(g, plane, b, h, t % g.ring));
    dst[vi] = src[vi];
  }
}

// ---------------------------------------------------------------------------
// Copy new tokens into the full-precision planes (blockIdx.y: 0 keys, 1
// values): FLOAT cache (slot t), KIVI residual ring (tokens t >= q1, slot
// t mod (R + G)), KVarN sinks (t < S, slot t) and staging ring (t >= S + n1 G,
// slot (t - S) mod G).  Always the final kernel of an append.
// ---------------------------------------------------------------------------
__global__ void store_full_kernel(Geom g, int L, const void* k, const void* v) {
  pdl_wait();
  pdl_trigger();
  bool ok;
  const int T0 = append_begin(g, L, &ok);
  const int T1 = T0 + L;
  if (ok) {
    const int which = blockIdx.y;
    const void* x = which ? v : k;
    const int es = g.act == KVQ_BF16 ? 2 : 4;
    const int vec_per_tok = g.D * es / 16;          // a power of two
    // the tokens that go to a full-precision plane: [a0, a1) and [c0, c1)
    int a0 = T0, a1 = T1, c0 = T1, c1 = T1;
    if (g.fmt == KVQ_FMT_KIVI) {
      a0 = max(T0, kivi_tq(T1, g.R, g.G));
    } else if (g.fmt == KVQ_FMT_KVARN) {
      const int pend_lo = g.S + kvarn_nblocks(T1, g.S, g.G) * g.G;
      a1 = max(T0, min(T1, g.S));
      c0 = min(max(T0, pend_lo), T1);
    }
    const int na = a1 - a0, n = na + (c1 - c0);
    const int total = g.B * g.H * n * vec_per_tok;   // below 2^31 (checked by the host)
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < total; i += gridDim.x * blockDim.x) {
      const int vi = i & (vec_per_tok - 1);
      const int rest = i / vec_per_tok;
      const int row = rest / n, j = rest - row * n;
      const int h = row % g.H, b = row / g.H;
      const int t = j < na ? a0 + j : c0 + (j - na);
      int plane, slot;
      if (g.fmt == KVQ_FMT_FLOAT) {
        plane = which ? KVQ_PLANE_V_FULL : KVQ_PLANE_K_FULL;
        slot = t;
      } else if (g.fmt == KVQ_FMT_KIVI) {
        plane = which ? KVQ_PLANE_V_FULL : KVQ_PLANE_K_FULL;
        slot = t % g.ring;
      } else if (t < g.S) {                       // KVarN sinks
        plane = which ? KVQ_PLANE_V_FULL : KVQ_PLANE_K_FULL;
        slot = t;
      } else {                                    // KVarN staging ring
        plane = which ? KVQ_PLANE_V_PEND : KVQ_PLANE_K_PEND;
        slot = (t - g.S) % g.G;
      }
      const uint4* src = reinterpret_cast<const uint4*>(
          reinterpret_cast<const char*>(x) + ((((int64_t)b * g.H + h) * L + (t - T0)) * g.D) * es);
      const Plane& pl = g.pl[plane];
      uint4* dst = reinterpret_cast<uint4*>(reinterpret_cast<char*>(pl.p) +
                                            plane_index(pl, b, h, g.H, slot, 0) * es);
      dst[vi] = src[vi];
    }
  }
  append_arrive_spread(g.state, T0, L, ok);
}

// ---------------------------------------------------------------------------
// KIVI keys: one group per (G-token block, channel).  One CTA per block that
// this append completes (grid sized for the most an append of L can flush):
// the block's G x D keys come in as 8-element vectors (residual ring or
// input) into shared memory, 256 / D threads per channel find partial min /
// max over their share of the G tokens, combine them and code their share,
// and each output word of a token's packed row is gathered from the byte
// codes and stored whole.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) kivi_key_flush_kernel(Geom g, int L, TokSrc src) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ float smem[];
  bool ok = true;
  const int T0u = g.layout == KVQ_LAYOUT_UNIFORM ? append_begin(g, L, &ok) : 0;
  const int G = g.G, D = g.D, bits = g.kb;
  int T0, n;
  append_span(g, blockIdx.y / g.H, L, T0u, &T0, &n);
  const int q0 = kivi_tq(T0, g.R, G), q1 = kivi_tq(T0 + n, g.R, G);
  const int blk = q0 / G + blockIdx.x;
  if (!ok || blk >= q1 / G) return;
  src.T0 = T0;
  float* xs = smem;                                   // [G][D]
  uint8_t* cs = reinterpret_cast<uint8_t*>(xs + G * D); // [G][D]
  const int h = blockIdx.y % g.H, b = blockIdx.y / g.H;
  const int t0 = blk * G;
  const int cpt = D / 8;
  for (int i = threadIdx.x; i < G * cpt; i += blockDim.x) {
    const int r = i / cpt, c8 = i - r * cpt;
    const void* sb;
    const int64_t e = tok_elem(g, src, b, h, t0 + r, &sb) + c8 * 8;
    float v[8];
    load8(sb, e, g.act, v);
    float4* dst = reinterpret_cast<float4*>(xs + r * D + c8 * 8);
    dst[0] = make_float4(v[0], v[1], v[2], v[3]);
    dst[1] = make_float4(v[4], v[5], v[6], v[7]);
  }
  __syncthreads();
  // parts threads per channel, each over G / parts tokens: partial min / max,
  // then every part codes its tokens with the channel's scale
  const int parts = (int)blockDim.x >= D ? (int)blockDim.x / D : 1;
  float* pmn = reinterpret_cast<float*>(cs + G * D);     // [parts][D]
  float* pmx = pmn + parts * D;
  for (int t = threadIdx.x; t < D * parts; t += blockDim.x) {
    const int d = t % D, part = t / D;
    const int r0 = part * G / parts, r1 = (part + 1) * G / parts;
    float mn = xs[r0 * D + d], mx = mn;
    for (int r = r0 + 1; r < r1; ++r) {
      mn = fminf(mn, xs[r * D + d]);
      mx = fmaxf(mx, xs[r * D + d]);
    }
    pmn[t] = mn;
    pmx[t] = mx;
  }
  __syncthreads();
  for (int t = threadIdx.x; t < D * parts; t += blockDim.x) {
    const int d = t % D, part = t / D;
    const int r0 = part * G / parts, r1 = (part + 1) * G / parts;
    float mn = pmn[d], mx = pmx[d];
    for (int p = 1; p < parts; ++p) {
      mn = fminf(mn, pmn[p * D + d]);
      mx = fmaxf(mx, pmx[p * D + d]);
    }
    const float s = affine_scale(mn, mx, bits), inv = __frcp_rn(s);
    bool ok = true;
    for (int r = r0; r < r1; ++r)
      cs[r * D + d] = (uint8_t)clamp_code(rint_quot_fast(__fsub_rn(xs[r * D + d], mn), inv, ok), bits);
    if (!ok)                                   // a quotient near a tie: all of them exactly
      for (int r = r0; r < r1; ++r)
        cs[r * D + d] = (uint8_t)affine_code(xs[r * D + d], mn, s, inv, bits);
    if (part == 0) {
      *blk_ptr<__half>(g, KVQ_PLANE_K_SCALE, b, h, blk, d) = __float2half_rn(s);
      *blk_ptr<__half>(g, KVQ_PLANE_K_ZERO, b, h, blk, d) = __float2half_rn(mn + 0.0f);
    }
  }
  __syncthreads();
  // 32-bit words of packed codes, LSB first: 32 / bits channels per word,
  // gathered from the byte codes with word loads and shifts
  const int cpw = 32 / bits, wpr = D / cpw;
  for (int i = threadIdx.x; i < G * wpr; i += blockDim.x) {
    const int r = i / wpr, w = i - r * wpr;
    const uint8_t* c = cs + r * D + w * cpw;
    uint32_t word;
    if (bits == 8) {
      word = *reinterpret_cast<const uint32_t*>(c);
    } else if (bits == 4) {                  // 4 bytes b0..b3 < 16 -> b0 | b1 << 4 | ...
      const uint2 u = *reinterpret_cast<const uint2*>(c);
      const uint32_t lo = u.x | (u.x >> 4), hi = u.y | (u.y >> 4);
      word = (lo & 0xFFu) | ((lo >> 8) & 0xFF00u) | ((hi & 0xFFu) << 16) | ((hi >> 8) & 0xFF00u) << 16;
    } else {                                 // 4 bytes b0..b3 < 4 -> b0 | b1 << 2 | ...
      const uint4 u = *reinterpret_cast<const uint4*>(c);
      auto crumbs = [](uint32_t q) {
        uint32_t t = q | (q >> 6);
        return (t | (t >> 12)) & 0xFFu;
      };
      word = crumbs(u.x) | crumbs(u.y) << 8 | crumbs(u.z) << 16 | crumbs(u.w) << 24;
    }
    reinterpret_cast<uint32_t*>(tok_ptr<uint8_t>(g, KVQ_PLANE_K_CODES, b, h, t0 + r))[w] = word;
  }
}

// The same flush for 32-token blocks with D and the bit width fixed at
// compile time (the KIVI configuration): 256 threads, 256 / D of them per
// channel over 32 D / 256 tokens each; codes go to shared memory as bytes and
// leave as whole packed words.  Same arithmetic as kivi_key_flush_kernel.
// One 32-token key block `blk` of the (b, h) row, by the CTA's 256 threads
// (src.T0 set: tokens below it come from the residual ring).
template <int D, int BITS>
__device__ __forceinline__ void kivi_key_flush32_block(const Geom& g, const TokSrc& src, int b,
                                                       int h, int blk, float* smem) {
  constexpr int G = 32, NT = 256, CPT = D / 8, PARTS = NT / D, TPP = G / PARTS;
  constexpr int CPW = 32 / BITS, WPR = D / CPW;
  float* xs = smem;                                      // [G][D]
  uint8_t* cs = reinterpret_cast<uint8_t*>(xs + G * D);  // [G][D]
  float* pmn = reinterpret_cast<float*>(cs + G * D);     // [PARTS][D]
  float* pmx = pmn + PARTS * D;
  const int t0 = blk * G;
#pragma unroll
  for (int k = 0; k < G * CPT / NT; ++k) {
    const int i = threadIdx.x + k * NT;
    const int r = i / CPT, c8 = i % CPT;
    const void* sb;
    const int64_t e = tok_elem(g, src, b, h, t0 + r, &sb) + c8 * 8;
    float v[8];
    load8(sb, e, g.act, v);
    float4* dst = reinterpret_cast<float4*>(xs + r * D + c8 * 8);
    dst[0] = make_float4(v[0], v[1], v[2], v[3]);
    dst[1] = make_float4(v[4], v[5], v[6], v[7]);
  }
  __syncthreads();
  const int d = threadIdx.x % D, part = threadIdx.x / D, r0 = part * TPP;
  float x[TPP];
  float mn, mx;
#pragma unroll
  for (int j = 0; j < TPP; ++j) x[j] = xs[(r0 + j) * D + d];
  mn = mx = x[0];
#pragma unroll
  for (int j = 1; j < TPP; ++j) {
    mn = fminf(mn, x[j]);
    mx = fmaxf(mx, x[j]);
  }
  pmn[threadIdx.x] = mn;
  pmx[threadIdx.x] = mx;
  __syncthreads();
  mn = pmn[d];
  mx = pmx[d];
#pragma unroll
  for (int p = 1; p < PARTS; ++p) {
    mn = fminf(mn, pmn[p * D + d]);
    mx = fmaxf(mx, pmx[p * D + d]);
  }
  const float s = affine_scale(mn, mx, BITS), inv = __frcp_rn(s);
  bool fast = true;
  float c[TPP];
#pragma unroll
  for (int j = 0; j < TPP; ++j) c[j] = rint_quot_fast(__fsub_rn(x[j], mn), inv, fast);
  if (!fast) {                                 // a quotient near a tie: all of them exactly
#pragma unroll
    for (int j = 0; j < TPP; ++j) c[j] = rintf(__fdiv_rn(__fsub_rn(x[j], mn), s));
  }
#pragma unroll
  for (int j = 0; j < TPP; ++j) cs[(r0 + j) * D + d] = (uint8_t)clamp_code(c[j], BITS);
  if (part == 0) {
    *blk_ptr<__half>(g, KVQ_PLANE_K_SCALE, b, h, blk, d) = __float2half_rn(s);
    *blk_ptr<__half>(g, KVQ_PLANE_K_ZERO, b, h, blk, d) = __float2half_rn(mn + 0.0f);
  }
  __syncthreads();
  for (int i = threadIdx.x; i < G * WPR; i += NT) {
    const int r = i / WPR, w = i % WPR;
    const uint8_t* cp = cs + r * D + w * CPW;
    uint32_t word;
    if (BITS == 8) {
      word = *reinterpret_cast<const uint32_t*>(cp);
    } else if (BITS == 4) {
      const uint2 u = *reinterpret_cast<const uint2*>(cp);
      const uint32_t lo = u.x | (u.x >> 4), hi = u.y | (u.y >> 4);
      word = (lo & 0xFFu) | ((lo >> 8) & 0xFF00u) | ((hi & 0xFFu) << 16) | ((hi >> 8) & 0xFF00u) << 16;
    } else {
      const uint4 u = *reinterpret_cast<const uint4*>(cp);
      auto crumbs = [](uint32_t q) {
        uint32_t t = q | (q >> 6);
        return (t | (t >> 12)) & 0xFFu;
      };
      word = crumbs(u.x) | crumbs(u.y) << 8 | crumbs(u.z) << 16 | crumbs(u.w) << 24;
    }
    reinterpret_cast<uint32_t*>(tok_ptr<uint8_t>(g, KVQ_PLANE_K_CODES, b, h, t0 + r))[w] = word;
  }
}

template <int D, int BITS>
__global__ void __launch_bounds__(256) kivi_key_flush32_kernel(Geom g, int L, TokSrc src) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ float smem[];
  bool ok = true;
  const int T0u = g.layout == KVQ_LAYOUT_UNIFORM ? append_begin(g, L, &ok) : 0;
  int T0, n;
  append_span(g, blockIdx.y / g.H, L, T0u, &T0, &n);
  const int q0 = kivi_tq(T0, g.R, 32), q1 = kivi_tq(T0 + n, g.R, 32);
  const int blk = q0 / 32 + blockIdx.x;
  if (!ok || blk >= q1 / 32) return;
  src.T0 = T0;
  kivi_key_flush32_block<D, BITS>(g, src, blockIdx.y / g.H, blockIdx.y % g.H, blk, smem);
}

// One decode token (L = 1) of a uniform KIVI cache with 32-token blocks, in
// one launch instead of three: one CTA per (b, h) codes the key block and
// the value tokens that this token completes (read from the residual ring,
// with the code of kivi_key_flush32_kernel and pack_pertoken_kernel), then
// stores the new key and value in the ring (as store_full_kernel does), and
// the last CTA advances the token count.  The block's ring slots and the new
// token's slot differ (the ring holds R + 32 tokens).
template <int D, int BITS>
__global__ void __launch_bounds__(256) kivi_decode_append_kernel(Geom g, const void* k,
                                                                 const void* v, int lcpt,
                                                                 int llpg) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ float smem[];
  bool ok = true;
  const int T0 = append_begin(g, 1, &ok);
  // grid (1, B H): pack_rows spreads a row's chunks over blockIdx.x
  const int b = blockIdx.y / g.H, h = blockIdx.y % g.H;
  const int q0 = kivi_tq(T0, g.R, 32), q1 = kivi_tq(T0 + 1, g.R, 32);
  if (ok && q1 > q0) {
    const TokSrc sk{k, T0, 1, KVQ_PLANE_K_FULL, 0, g.ring};
    kivi_key_flush32_block<D, BITS>(g, sk, b, h, q0 / 32, smem);
    const TokSrc sv{v, T0, 1, KVQ_PLANE_V_FULL, 0, g.ring};
    pack_rows(g, sv, b, h, q0, q1 - q0, 1, 0, lcpt, llpg);
  }
  if (ok && T0 >= q1) {                      // the new token stays in full precision
    constexpr int V16 = D * 2 / 16;          // 16-byte pieces of a bf16 row
    if ((int)threadIdx.x < 2 * V16) {
      const int which = threadIdx.x / V16, vi = threadIdx.x % V16;
      const int plane = which ? KVQ_PLANE_V_FULL : KVQ_PLANE_K_FULL;
      const uint4* src = reinterpret_cast<const uint4*>(which ? v : k) +
                         ((int64_t)b * g.H + h) * V16;
      const Plane& pl = g.pl[plane];
      uint4* dst = reinterpret_cast<uint4*>(reinterpret_cast<char*>(pl.p) +
                                            plane_index(pl, b, h, g.H, T0 % g.ring, 0) * 2);
      dst[vi] = src[vi];
    }
  }
  append_arrive_spread(g.state, T0, 1, ok);
}

// ---------------------------------------------------------------------------
// KVarN block: normalised Hadamard on D, dual-axis variance normalisation,
// grouped affine along D.  One CTA per (block this append completes, b*h,
// k|v).  Sums follow the stride-halving pairwise tree in fp32.
// ---------------------------------------------------------------------------
__global__ void kvarn_block_kernel(Geom g, int L, TokSrc sk, TokSrc sv, float inv_sqrt_d) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ float smem[];
  bool ok;
  const int T0 = append_begin(g, L, &ok);
  const int G = g.G, D = g.D;
  const int n0 = kvarn_nblocks(T0, g.S, G), n1 = kvarn_nblocks(T0 + L, g.S, G);
  const int blk = n0 + blockIdx.x;
  if (!ok || blk >= n1) return;
  const int which = blockIdx.z;
  TokSrc src = which ? sv : sk;
  src.T0 = T0;
  const int bits = which ? g.vb : g.kb;
  float* y = smem;                 // [G][D]
  float* acc = y + G * D;          // [G][D] scratch for the sums, then codes
  float* sig = acc + G * D;        // [max(G, D)]
  float* rsc = sig + 256;          // [G] row scales
  float* csc = rsc + 128;          // [D] column scales
  const int h = blockIdx.y % g.H, b = blockIdx.y / g.H;
  const int q0 = blk * G;          // first quantized row of the block
  const int t0 = g.S + q0;
  const int nt = blockDim.x;
  for (int i = threadIdx.x; i < G * D; i += nt) {
    const int r = i / D, d = i % D;
    const void* sb;
    int64_t e = tok_elem(g, src, b, h, t0 + r, &sb);
    y[i] = ld_act(sb, e + d, g.act);
  }
  for (int i = threadIdx.x; i < G; i += nt) rsc[i] = 1.f;
  for (int i = threadIdx.x; i < D; i += nt) csc[i] = 1.f;
  __syncthreads();
  // Hadamard butterflies, h = 1, 2, ..., D/2
  for (int hs = 1; hs < D; hs <<= 1) {
    for (int p = threadIdx.x; p < G * D / 2; p += nt) {
      const int r = p / (D / 2), k = p % (D / 2);
      const int j = (k / hs) * 2 * hs + (k % hs);
      float a = y[r * D + j], c = y[r * D + j + hs];
      y[r * D + j] = __fadd_rn(a, c);
      y[r * D + j + hs] = __fsub_rn(a, c);
    }
    __syncthreads();
  }
  for (int i = threadIdx.x; i < G * D; i += nt) y[i] = __fmul_rn(y[i], inv_sqrt_d);
  __syncthreads();
  const float inv_d = 1.f / (float)D, inv_g = 1.f / (float)G;
  for (int it = 0; it < g.iters; ++it) {
    // rows
    for (int i = threadIdx.x; i < G * D; i += nt) acc[i] = __fmul_rn(y[i], y[i]);
    __syncthreads();
    for (int n = D / 2; n >= 1; n >>= 1) {
      for (int p = threadIdx.x; p < G * n; p += nt) {
        const int r = p / n, j = p % n;
        acc[r * D + j] = __fadd_rn(acc[r * D + j], acc[r * D + j + n]);
      }
      __syncthreads();
    }
    for (int r = threadIdx.x; r < G; r += nt) {
      const float sg = fmaxf(__fsqrt_rn(__fmul_rn(acc[r * D], inv_d)), 1e-8f);
      sig[r] = sg;
      rsc[r] = __fmul_rn(rsc[r], sg);
    }
    __syncthreads();
    for (int i = threadIdx.x; i < G * D; i += nt) y[i] = __fdiv_rn(y[i], sig[i / D]);
    __syncthreads();
    // columns
    for (int i = threadIdx.x; i < G * D; i += nt) acc[i] = __fmul_rn(y[i], y[i]);
    __syncthreads();
    for (int n = G / 2; n >= 1; n >>= 1) {
      for (int p = threadIdx.x; p < n * D; p += nt) {
        const int r = p / D, j = p % D;
        acc[r * D + j] = __fadd_rn(acc[r * D + j], acc[(r + n) * D + j]);
      }
      __syncthreads();
    }
    for (int j = threadIdx.x; j < D; j += nt) {
      const float sg = fmaxf(__fsqrt_rn(__fmul_rn(acc[j], inv_g)), 1e-8f);
      sig[j] = sg;
      csc[j] = __fmul_rn(csc[j], sg);
    }
    __syncthreads();
    for (int i = threadIdx.x; i < G * D; i += nt) y[i] = __fdiv_rn(y[i], sig[i % D]);
    __syncthreads();
  }
  // grouped affine along D (groups of G channels)
  const int codes_plane = which ? KVQ_PLANE_V_CODES : KVQ_PLANE_K_CODES;
  const int scale_plane = which ? KVQ_PLANE_V_SCALE : KVQ_PLANE_K_SCALE;
  const int zero_plane = which ? KVQ_PLANE_V_ZERO : KVQ_PLANE_K_ZERO;
  const int row_plane = which ? KVQ_PLANE_V_ROW : KVQ_PLANE_K_ROW;
  const int col_plane = which ? KVQ_PLANE_V_COL : KVQ_PLANE_K_COL;
  uint8_t* cs = reinterpret_cast<uint8_t*>(acc);
  const int ng = D / G;
  for (int p = threadIdx.x; p < G * ng; p += nt) {
    const int r = p / ng, gq = p % ng;
    const float* row = y + r * D + gq * G;
    float mn = row[0], mx = row[0];
    for (int j = 1; j < G; ++j) { mn = fminf(mn, row[j]); mx = fmaxf(mx, row[j]); }
    const float sc = affine_scale(mn, mx, bits), inv = __frcp_rn(sc);
    bool ok = true;
    for (int j = 0; j < G; ++j)
      cs[r * D + gq * G + j] = (uint8_t)clamp_code(rint_quot_fast(__fsub_rn(row[j], mn), inv, ok), bits);
    if (!ok)                                   // a quotient near a tie: all of them exactly
      for (int j = 0; j < G; ++j)
        cs[r * D + gq * G + j] = (uint8_t)affine_code(row[j], mn, sc, inv, bits);
    *plane_ptr<__half>(g, scale_plane, b, h, q0 + r, gq) = __float2half_rn(sc);
    *plane_ptr<__half>(g, zero_plane, b, h, q0 + r, gq) = __float2half_rn(mn + 0.0f);
  }
  for (int r = threadIdx.x; r < G; r += nt)
    *plane_ptr<__half>(g, row_plane, b, h, 0, q0 + r) = __float2half_rn(rsc[r]);
  for (int j = threadIdx.x; j < D; j += nt)
    *plane_ptr<__half>(g, col_plane, b, h, blk, j) = __float2half_rn(csc[j]);
  __syncthreads();
  const int per = 8 / bits, row_bytes = D * bits / 8;
  for (int i = threadIdx.x; i < G * row_bytes; i += nt) {
    const int r = i / row_bytes, j = i % row_bytes;
    unsigned byte = 0;
    for (int e = 0; e < per; ++e) byte |= (unsigned)cs[r * D + j * per + e] << (e * bits);
    plane_ptr<uint8_t>(g, codes_plane, b, h, q0 + r)[j] = (uint8_t)byte;
  }
}

// The same block transform with warps instead of CTA-wide steps (D = 64/128/
// 256, G = 32/64).  Every floating-point operation and its order are those of
// kvarn_block_kernel (and of the reference definition): Hadamard stages
// h = 1 .. D/2 with explicit fp32 add/sub, the stride-halving pairwise trees
// for the row and column sums of squares, IEEE sqrt and division.  A warp
// owns whole rows for the Hadamard and the row statistics (lane l holds
// channels l + 32 i: the upper tree levels add slots in registers, the last
// five add lanes by xor-shuffle); a thread owns a whole column for the column
// statistics (the tree in registers).  Two CTA barriers per iteration.
template <int D, int G>
__global__ void __launch_bounds__(256)
kvarn_block_fast_kernel(Geom g, int L, TokSrc sk, TokSrc sv, float inv_sqrt_d) {
  pdl_wait();
  pdl_trigger();
  constexpr int NS = D / 32, NG = D / G;
  extern __shared__ float smem[];
  bool ok;
  const int T0 = append_begin(g, L, &ok);
  const int n0 = kvarn_nblocks(T0, g.S, G), n1 = kvarn_nblocks(T0 + L, g.S, G);
  const int blk = n0 + blockIdx.x;
  if (!ok || blk >= n1) return;
  const int which = blockIdx.z;
  TokSrc src = which ? sv : sk;
  src.T0 = T0;
  const int bits = which ? g.vb : g.kb;
  float* y = smem;                                // [G][D]
  float* rsc = y + G * D;                         // [G] row scales
  float* csc = rsc + G;                           // [D] column scales
  uint8_t* cs = reinterpret_cast<uint8_t*>(csc + D);   // [G][D] codes
  const int h = blockIdx.y % g.H, b = blockIdx.y / g.H;
  const int q0 = blk * G, t0 = g.S + q0;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // load and rotate: a warp per row
  for (int r = warp; r < G; r += 8) {
    float x[NS];
    const void* sb;
    const int64_t e = tok_elem(g, src, b, h, t0 + r, &sb);
#pragma unroll
    for (int i = 0; i < NS; ++i) x[i] = ld_act(sb, e + lane + 32 * i, g.act);
#pragma unroll
    for (int hh = 1; hh < 32; hh <<= 1)
#pragma unroll
      for (int i = 0; i < NS; ++i) {
        const float o = __shfl_xor_sync(0xffffffffu, x[i], hh);
        x[i] = (lane & hh) ? __fsub_rn(o, x[i]) : __fadd_rn(x[i], o);
      }
#pragma unroll
    for (int hs = 1; hs < NS; hs <<= 1)
#pragma unroll
      for (int i = 0; i < NS; ++i)
        if (!(i & hs)) {
          const float a = x[i], c = x[i + hs];
          x[i] = __fadd_rn(a, c);
          x[i + hs] = __fsub_rn(a, c);
        }
#pragma unroll
    for (int i = 0; i < NS; ++i) y[r * D + lane + 32 * i] = __fmul_rn(x[i], inv_sqrt_d);
    if (lane == 0) rsc[r] = 1.f;
  }
  for (int j = threadIdx.x; j < D; j += blockDim.x) csc[j] = 1.f;
  __syncthreads();
  const float inv_d = 1.f / (float)D, inv_g = 1.f / (float)G;
  for (int it = 0; it < g.iters; ++it) {
    // rows
    for (int r = warp; r < G; r += 8) {
      float x[NS], a[NS];
#pragma unroll
      for (int i = 0; i < NS; ++i) {
        x[i] = y[r * D + lane + 32 * i];
        a[i] = __fmul_rn(x[i], x[i]);
      }
#pragma unroll
      for (int ns = NS / 2; ns >= 1; ns >>= 1)
#pragma unroll
        for (int i = 0; i < ns; ++i) a[i] = __fadd_rn(a[i], a[i + ns]);
#pragma unroll
      for (int n = 16; n >= 1; n >>= 1) a[0] = __fadd_rn(a[0], __shfl_xor_sync(0xffffffffu, a[0], n));
      const float sum = __shfl_sync(0xffffffffu, a[0], 0);
      const float sg = fmaxf(__fsqrt_rn(__fmul_rn(sum, inv_d)), 1e-8f);
      if (lane == 0) rsc[r] = __fmul_rn(rsc[r], sg);
#pragma unroll
      for (int i = 0; i < NS; ++i) y[r * D + lane + 32 * i] = __fdiv_rn(x[i], sg);
    }
    __syncthreads();
    // columns: a thread per column
    for (int j = threadIdx.x; j < D; j += blockDim.x) {
      float col[G], a[G];
#pragma unroll
      for (int r = 0; r < G; ++r) {
        col[r] = y[r * D + j];
        a[r] = __fmul_rn(col[r], col[r]);
      }
#pragma unroll
      for (int n = G / 2; n >= 1; n >>= 1)
#pragma unroll
        for (int r = 0; r < n; ++r) a[r] = __fadd_rn(a[r], a[r + n]);
      const float sg = fmaxf(__fsqrt_rn(__fmul_rn(a[0], inv_g)), 1e-8f);
      csc[j] = __fmul_rn(csc[j], sg);
#pragma unroll
      for (int r = 0; r < G; ++r) y[r * D + j] = __fdiv_rn(col[r], sg);
    }
    __syncthreads();
  }
  // grouped affine along D (groups of G channels)
  const int codes_plane = which ? KVQ_PLANE_V_CODES : KVQ_PLANE_K_CODES;
  const int scale_plane = which ? KVQ_PLANE_V_SCALE : KVQ_PLANE_K_SCALE;
  const int zero_plane = which ? KVQ_PLANE_V_ZERO : KVQ_PLANE_K_ZERO;
  const int row_plane = which ? KVQ_PLANE_V_ROW : KVQ_PLANE_K_ROW;
  const int col_plane = which ? KVQ_PLANE_V_COL : KVQ_PLANE_K_COL;
  // a thread per (row, group); each lane walks its group from its own lane
  // offset, so the lanes of a warp read (and write) different banks (min, max
  // and the codes do not depend on the order)
  const int rot = threadIdx.x & 31;
  for (int p = threadIdx.x; p < G * NG; p += blockDim.x) {
    const int r = p / NG, gq = p % NG;
    const float* row = y + r * D + gq * G;
    uint8_t* crow = cs + r * D + gq * G;
    float mn = row[rot & (G - 1)], mx = mn;
    for (int jj = 1; jj < G; ++jj) {
      const float x = row[(jj + rot) & (G - 1)];
      mn = fminf(mn, x);
      mx = fmaxf(mx, x);
    }
    const float sc = affine_scale(mn, mx, bits), inv = __frcp_rn(sc);
    bool ok = true;
    for (int jj = 0; jj < G; ++jj) {
      const int j = (jj + rot) & (G - 1);
      crow[j] = (uint8_t)clamp_code(rint_quot_fast(__fsub_rn(row[j], mn), inv, ok), bits);
    }
    if (!ok)                                   // a quotient near a tie: all of them exactly
      for (int j = 0; j < G; ++j) crow[j] = (uint8_t)affine_code(row[j], mn, sc, inv, bits);
    *plane_ptr<__half>(g, scale_plane, b, h, q0 + r, gq) = __float2half_rn(sc);
    *plane_ptr<__half>(g, zero_plane, b, h, q0 + r, gq) = __float2half_rn(mn + 0.0f);
  }
  for (int r = threadIdx.x; r < G; r += blockDim.x)
    *plane_ptr<__half>(g, row_plane, b, h, 0, q0 + r) = __float2half_rn(rsc[r]);
  for (int j = threadIdx.x; j < D; j += blockDim.x)
    *plane_ptr<__half>(g, col_plane, b, h, blk, j) = __float2half_rn(csc[j]);
  __syncthreads();
  const int per = 8 / bits, row_bytes = D * bits / 8;
  for (int i = threadIdx.x; i < G * row_bytes; i += blockDim.x) {
    const int r = i / row_bytes, j = i % row_bytes;
    unsigned byte = 0;
    for (int e = 0; e < per; ++e) byte |= (unsigned)cs[r * D + j * per + e] << (e * bits);
    plane_ptr<uint8_t>(g, codes_plane, b, h, q0 + r)[j] = (uint8_t)byte;
  }
}

template <int D, int G>
cudaError_t launch_kvarn_fast(const Geom& g, int max_blocks, int L, const TokSrc& sk,
                              const TokSrc& sv, float inv_sqrt_d, cudaStream_t s) {
  const size_t sm = (size_t)G * D * 4 + (size_t)(G + D) * 4 + (size_t)G * D;
  auto kern = kvarn_block_fast_kernel<D, G>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
  if (e != cudaSuccess) return e;
  launch_pdl(kern, dim3(dim3(max_blocks, g.B * g.H, 2)), dim3(256), sm, s, g, L, sk, sv, inv_sqrt_d);
  return cudaGetLastError();
}

cudaError_t launch_kvarn_blocks(const Geom& g, int max_blocks, int L, const TokSrc& sk,
                                const TokSrc& sv, float inv_sqrt_d, cudaStream_t s) {
  if (g.G == 32) {
    if (g.D == 64) return launch_kvarn_fast<64, 32>(g, max_blocks, L, sk, sv, inv_sqrt_d, s);
    if (g.D == 128) return launch_kvarn_fast<128, 32>(g, max_blocks, L, sk, sv, inv_sqrt_d, s);
    if (g.D == 256) return launch_kvarn_fast<256, 32>(g, max_blocks, L, sk, sv, inv_sqrt_d, s);
  } else if (g.G == 64) {
    if (g.D == 64) return launch_kvarn_fast<64, 64>(g, max_blocks, L, sk, sv, inv_sqrt_d, s);
    if (g.D == 128) return launch_kvarn_fast<128, 64>(g, max_blocks, L, sk, sv, inv_sqrt_d, s);
    if (g.D == 256) return launch_kvarn_fast<256, 64>(g, max_blocks, L, sk, sv, inv_sqrt_d, s);
  }
  return cudaErrorNotSupported;
}

// Grid of the per-token coder: (chunk blocks of a row, B H rows, keys |
// values), x capped so the whole grid stays within 8 CTAs per SM.
dim3 pertoken_grid(const Geom& g, int ntok_max, int which_count) {
  const int64_t chunks = (int64_t)ntok_max * (g.D / 8);
  int64_t gx = (chunks + 255) / 256;
  const int64_t cap = (int64_t)num_sms() * 8 / ((int64_t)g.B * g.H * which_count);
  if (gx > cap) gx = cap;
  if (gx < 1) gx = 1;
  return dim3((unsigned)gx, (unsigned)(g.B * g.H), (unsigned)which_count);
}

int ilog2(int x) {
  int l = 0;
  while ((1 << (l + 1)) <= x) ++l;
  return l;
}

int grid_for(int64_t threads_needed, int block) {
  int64_t n = (threads_needed + block - 1) / block;
  int64_t cap = (int64_t)num_sms() * 8;
  if (n > cap) n = cap;
  return (int)(n < 1 ? 1 : n);
}

// KIVI: code the key blocks and the value blocks this append completes
// (before the ring takes the new tokens: the blocks read older tokens from it).
cudaError_t launch_kivi_append(const Geom& g, int L, const void* k, const void* v,
                               cudaStream_t s) {
  TokSrc sk{k, 0, L, KVQ_PLANE_K_FULL, 0, g.ring}, sv{v, 0, L, KVQ_PLANE_V_FULL, 0, g.ring};
  const int max_blocks = L / g.G + 1;     // most G-blocks an append of L completes
  const size_t sm = (size_t)g.G * g.D * 5 + 2 * 256 * sizeof(float);
  cudaError_t e = cudaFuncSetAttribute(kivi_key_flush_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
  if (e != cudaSuccess) return e;
  const dim3 fgrid(max_blocks, g.B * g.H);
  auto fk = kivi_key_flush_kernel;
  if (g.G == 32) {
    const int b = g.kb;
    if (g.D == 64) fk = b == 2 ? kivi_key_flush32_kernel<64, 2> : b == 4 ? kivi_key_flush32_kernel<64, 4> : kivi_key_flush32_kernel<64, 8>;
    if (g.D == 128) fk = b == 2 ? kivi_key_flush32_kernel<128, 2> : b == 4 ? kivi_key_flush32_kernel<128, 4> : kivi_key_flush32_kernel<128, 8>;
    if (g.D == 256) fk = b == 2 ? kivi_key_flush32_kernel<256, 2> : b == 4 ? kivi_key_flush32_kernel<256, 4> : kivi_key_flush32_kernel<256, 8>;
  }
  if (fk != kivi_key_flush_kernel) {
    e = cudaFuncSetAttribute(fk, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e != cudaSuccess) return e;
  }
  launch_pdl(fk, fgrid, dim3(256), sm, s, g, L, sk);
  launch_pdl(pack_pertoken_kernel, pertoken_grid(g, max_blocks * g.G, 1), dim3(256), 0, s, g,
             L, sk, sv, 0, 1, 0, ilog2(g.D / 8), ilog2(g.G / 8));
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_append_ragged(const Geom& g, int L, const void* k, const void* v,
                                 const int* n, cudaStream_t s) {
  SeqCounts c = {};
  for (int b = 0; b < g.B; ++b) c.n[b] = n[b];
  launch_pdl(seq_counts_kernel, dim3(1), dim3(256), 0, s, g, c);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if (g.fmt == KVQ_FMT_KIVI) {
    e = launch_kivi_append(g, L, k, v, s);
    if (e != cudaSuccess) return e;
    launch_pdl(store_ring_ragged_kernel,
               dim3(dim3(grid_for((int64_t)g.B * g.H * L * (g.D * 2 / 16), 256), 2)), dim3(256),
               0, s, g, L, k, v);
  } else {
    TokSrc sk{k, 0, L, -1, 0, 1}, sv{v, 0, L, -1, 0, 1};
    launch_pdl(pack_pertoken_kernel, pertoken_grid(g, L, 2), dim3(256), 0, s, g, L, sk, sv,
               g.fmt == KVQ_FMT_SYMMETRIC ? 1 : 0, 0, 0, ilog2(g.D / 8), ilog2(g.G / 8));
  }
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  launch_pdl(seq_advance_kernel, dim3(1), dim3(256), 0, s, g);
  return cudaGetLastError();
}

// A sequence of a ragged cache becomes empty.
__global__ void seq_reset_kernel(Geom g, int b) {
  pdl_wait();
  pdl_trigger();
  if (threadIdx.x == 0) {
    g.seq_len[b] = 0;
    g.seq_new[b] = 0;
  }
}

cudaError_t launch_seq_reset(const Geom& g, int b, cudaStream_t s) {
  launch_pdl(seq_reset_kernel, dim3(1), dim3(32), 0, s, g, b);
  return cudaGetLastError();
}

cudaError_t launch_append(const Geom& g, int L, const void* k, const void* v, cudaStream_t s) {
  TokSrc sk{k, 0, L, -1, 0, 1}, sv{v, 0, L, -1, 0, 1};
  const int es = g.act == KVQ_BF16 ? 2 : 4;
  const int64_t full_threads = (int64_t)g.B * g.H * L * (g.D * es / 16);
  const int max_blocks = L / g.G + 1;     // most G-blocks an append of L completes
  cudaError_t e;
  switch (g.fmt) {
    case KVQ_FMT_FLOAT:
      launch_pdl(store_full_kernel, dim3(dim3(grid_for(full_threads, 256), 2)), dim3(256), 0, s, g, L, k, v);
      return cudaGetLastError();
    case KVQ_FMT_AFFINE:
    case KVQ_FMT_SYMMETRIC: {
      const int sym = g.fmt == KVQ_FMT_SYMMETRIC;
      launch_pdl(pack_pertoken_kernel, pertoken_grid(g, L, 2), dim3(256), 0, s, g, L, sk, sv, sym,
                 0, 1, ilog2(g.D / 8), ilog2(g.G / 8));
      return cudaGetLastError();
    }
    case KVQ_FMT_KIVI: {
      if (L == 1 && g.G == 32 && g.act == KVQ_BF16 && g.kb == g.vb &&
          (g.D == 64 || g.D == 128 || g.D == 256) && (g.kb == 2 || g.kb == 4 || g.kb == 8)) {
        // a decode token: one launch
        auto kern = kivi_decode_append_kernel<128, 2>;
        if (g.D == 64) kern = g.kb == 2 ? kivi_decode_append_kernel<64, 2> : g.kb == 4 ? kivi_decode_append_kernel<64, 4> : kivi_decode_append_kernel<64, 8>;
        if (g.D == 128) kern = g.kb == 2 ? kivi_decode_append_kernel<128, 2> : g.kb == 4 ? kivi_decode_append_kernel<128, 4> : kivi_decode_append_kernel<128, 8>;
        if (g.D == 256) kern = g.kb == 2 ? kivi_decode_append_kernel<256, 2> : g.kb == 4 ? kivi_decode_append_kernel<256, 4> : kivi_decode_append_kernel<256, 8>;
        const size_t sm = (size_t)32 * g.D * 5 + 2 * 256 * sizeof(float);
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
        if (e != cudaSuccess) return e;
        launch_pdl(kern, dim3(1, g.B * g.H), dim3(256), sm, s, g, k, v, ilog2(g.D / 8), ilog2(32 / 8));
        return cudaGetLastError();
      }
      e = launch_kivi_append(g, L, k, v, s);
      if (e != cudaSuccess) return e;
      launch_pdl(store_full_kernel, dim3(dim3(grid_for(full_threads, 256), 2)), dim3(256), 0, s, g, L, k, v);
      return cudaGetLastError();
    }
    case KVQ_FMT_KVARN: {
      const size_t sm = ((size_t)2 * g.G * g.D + 256 + 128 + 256) * sizeof(float);
      const float inv_sqrt_d = (float)(1.0 / sqrt((double)g.D));
      e = cudaFuncSetAttribute(kvarn_block_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               (int)sm);
      if (e != cudaSuccess) return e;
      sk.ring_plane = KVQ_PLANE_K_PEND; sk.ring_off = g.S; sk.ring_rows = g.G;
      sv.ring_plane = KVQ_PLANE_V_PEND; sv.ring_off = g.S; sv.ring_rows = g.G;
      e = launch_kvarn_blocks(g, max_blocks, L, sk, sv, inv_sqrt_d, s);
      if (e == cudaErrorNotSupported) {
        (void)cudaGetLastError();
        launch_pdl(kvarn_block_kernel, dim3(dim3(max_blocks, g.B * g.H, 2)), dim3(256), sm, s, g, L, sk, sv, inv_sqrt_d);
      } else if (e != cudaSuccess) {
        return e;
      }
      launch_pdl(store_full_kernel, dim3(dim3(grid_for(full_threads, 256), 2)), dim3(256), 0, s, g, L, k, v);
      return cudaGetLastError();
    }
  }
  return cudaErrorInvalidValue;
}

}  // namespace kvq
