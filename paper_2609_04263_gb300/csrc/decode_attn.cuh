// Device code of the split-K decode attention (shared by the standalone
// kernel in attend_mma.cu and the fused decode step in decode_step.cu).
#pragma once

#include <math.h>

#include "kvq_internal.cuh"

namespace kvq {
namespace dattn {
// Split-K flash-decode over the packed cache on tensor cores (bf16 mma.sync).
//
// One CTA = (split of the tokens, kv head, sequence); 4 warps.  Each CTA
// writes its split's partial (m, l, o) to the workspace; the last CTA of a
// (sequence, kv head) to finish (an arrival counter, no waiting) merges them
// by log-sum-exp into the output.  The split's
// tokens stream through shared memory in 64-token chunks: one thread issues
// TMA bulk copies (codes and fp16 metadata of the chunk) on an mbarrier ring
// of kStages buffers; each warp then takes one 16-token tile of the chunk.
//
// Scores: S[h][t] = sum_d q[h][d] k_hat[t][d] with the g = Hq/Hkv query heads
// of the kv head as the MMA rows (zero-padded to 16) and tokens as columns.
// Codes enter the MMA as exact bf16 integers: (0x4300 | c) is the bf16 value
// 128 + c, built two at a time by one LOP3.  With per-token groups,
//   q . k_hat = sum_groups s_g (q_g . (c_g + 128)) + (m_g - 128 s_g) sum(q_g),
// so each group keeps its own accumulator and the scale and offset are applied
// per token after the MMA.  KIVI keys (one scale per block and channel) fold
// the scale into q instead: q' = q * s_blk, split into bf16 hi + lo.  Values
// run through fp16 MMAs with codes as (0x6400 | c) = 1024 + c:
//   O[h][d] += sum_t fp16(p s)[h][t] (c + 1024)[t][d] + sum_t (p m - 1024 fp16(p s)).
//
// The MMA's k index may map to any channel as long as q and k agree, and its
// output columns to any channel as long as the store undoes it; the mappings
// below make each thread's codes one contiguous word per group.

constexpr int kCT = 64;          // tokens per chunk (4 tiles of 16)
constexpr int kStages = 4;
constexpr int kWarps = 4;
constexpr uint32_t kMagic = 0x43004300u;
constexpr long kWaitLimit = 1L << 24;   // polls of an mbarrier before a wait gives up at the latest

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_inval(uint64_t* bar) {
  asm volatile("mbarrier.inval.shared::cta.b64 [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, int count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count));
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok) : "r"(smem_u32(bar)), "r"(parity) : "memory");
  return ok != 0;
}
// Wait bounded in time (try_wait may suspend the thread between polls, so a
// count of polls alone does not bound it); returns false (and the caller
// flags an error) after about a second.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  uint64_t t0;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t0));
  for (long i = 0;; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 7) == 7) {
      uint64_t t;
      asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
      if (t - t0 > 1000000000ull || i > kWaitLimit) return false;
    }
  }
}
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes,
                                         uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
      ::"r"(smem_u32(dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar)) : "memory");
}

// Tagged words: a float in the low half, the writer's launch tag in the high
// half, stored and loaded as one 64-bit access, so a reader that sees its own
// launch's tag also sees that launch's value (no fence or flag needed).
constexpr long kPollLimit = 1L << 20;   // polls of one L2 round trip: about a second
__device__ __forceinline__ void st_tagged(uint64_t* p, float v, uint32_t tag) {
  const uint64_t w = (uint64_t)__float_as_uint(v) | ((uint64_t)tag << 32);
  asm volatile("st.relaxed.gpu.global.b64 [%0], %1;" ::"l"(p), "l"(w) : "memory");
}
__device__ __forceinline__ uint64_t ld_tagged(const uint64_t* p) {
  uint64_t w;
  asm volatile("ld.relaxed.gpu.global.b64 %0, [%1];" : "=l"(w) : "l"(p) : "memory");
  return w;
}
// two adjacent tagged words (16-byte aligned) in one access
__device__ __forceinline__ void ld_tagged2(const uint64_t* p, uint64_t& a, uint64_t& b) {
  asm volatile("ld.relaxed.gpu.global.v2.b64 {%0, %1}, [%2];" : "=l"(a), "=l"(b) : "l"(p) : "memory");
}
__device__ __forceinline__ float tagged_value(uint64_t w) { return __uint_as_float((uint32_t)w); }
__device__ __forceinline__ bool tag_is(uint64_t w, uint32_t tag) { return (uint32_t)(w >> 32) == tag; }

__device__ __forceinline__ void mma16816(float c[4], const uint32_t a[4], uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
// (x & mask) | 0x43004300: two codes as bf16 (128 + c)
__device__ __forceinline__ uint32_t magic2(uint32_t x, uint32_t mask) {
  uint32_t r;
  asm("lop3.b32 %0, %1, %2, %3, 0xEA;" : "=r"(r) : "r"(x), "r"(mask), "r"(kMagic));
  return r;
}
// (x & mask) | 0x64006400: two codes as fp16 (1024 + c)
constexpr uint32_t kMagicH = 0x64006400u;
__device__ __forceinline__ uint32_t magic2h(uint32_t x, uint32_t mask) {
  uint32_t r;
  asm("lop3.b32 %0, %1, %2, %3, 0xEA;" : "=r"(r) : "r"(x), "r"(mask), "r"(kMagicH));
  return r;
}
__device__ __forceinline__ void mma16816_f16(float c[4], const uint32_t a[4], uint32_t b0,
                                             uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack_f16(float lo, float hi) {
  __half2 v = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}
__device__ __forceinline__ uint32_t pack_raw(uint16_t lo, uint16_t hi) {
  return (uint32_t)lo | ((uint32_t)hi << 16);
}

// Channel held by slot e (0..7) of a thread's 8-channel word in QK k-step s,
// register half (0: a0/b0, 1: a2/b1), element j: see the LOP3 pairings.
template <int BITS>
__device__ __forceinline__ int qk_chan(int s, int half, int j) {
  if (BITS == 4) return 2 * s + half + 4 * j;     // pairs (n0,n4),(n1,n5),(n2,n6),(n3,n7)
  return 4 * s + 2 * half + j;                     // pairs (c0,c1),(c2,c3),(c4,c5),(c6,c7)
}

template <int D, int BITS, int FMT>
struct Cfg {
  static constexpr int NG = D / 32;                 // quantization groups (G = 32)
  static constexpr int KSTEP = D / 16;
  static constexpr int CODE_B = D * BITS / 8;       // code bytes per token
  static constexpr int NT_PV = D / 8;               // PV n-tiles
  // shared memory per stage
  static constexpr int KC_OFF = 0;
  static constexpr int VC_OFF = KC_OFF + kCT * CODE_B;
  static constexpr int KS_OFF = VC_OFF + kCT * CODE_B;            // K scale (per token or block)
  static constexpr int KMETA_B = FMT == KVQ_FMT_KIVI ? (kCT / 32) * D * 2 : kCT * NG * 2;
  static constexpr int KZ_OFF = KS_OFF + KMETA_B;
  static constexpr int VS_OFF = KZ_OFF + KMETA_B;
  static constexpr int VZ_OFF = VS_OFF + kCT * NG * 2;
  static constexpr int STAGE_B = ((VZ_OFF + kCT * NG * 2) + 127) / 128 * 128;
};

// Token range of one split: [ts, te), coded tokens [0, tq), chunks of kCT.
struct SplitPlan {
  int ts, te, tq, nchunks;
};
template <int FMT>
__device__ __forceinline__ SplitPlan split_plan(const Geom& g, int T, int splits, int split) {
  SplitPlan p;
  split_range(T, splits, split, kCT, &p.ts, &p.te);
  p.tq = FMT == KVQ_FMT_KIVI ? kivi_tq(T, g.R, 32) : T;
  p.nchunks = p.te > p.ts ? (p.te - p.ts + kCT - 1) / kCT : 0;
  return p;
}

// Copies of one chunk (codes and fp16 metadata) into stage chunk % STAGES.
// One thread calls it.
template <int D, int BITS, int FMT, int STAGES>
__device__ void split_issue(const Geom& g, int b, int hkv, const SplitPlan& sp, int chunk,
                            unsigned char* smem, uint64_t* bars) {
  using C = Cfg<D, BITS, FMT>;
  constexpr int NG = C::NG;
  const int stage = chunk % STAGES;
  unsigned char* st = smem + stage * C::STAGE_B;
  const int c0 = sp.ts + chunk * kCT;
  int nq = min(kCT, sp.tq - c0);              // coded tokens of the chunk
  if (nq <= 0) {                              // nothing coded: arrive with no bytes
    mbar_expect_tx(&bars[stage], 0);
    return;
  }
  nq = (nq + 3) & ~3;                         // 16-byte multiples (planes padded)
  const uint32_t code_bytes = nq * C::CODE_B;
  const uint32_t kmeta = FMT == KVQ_FMT_KIVI ? ((nq + 31) / 32) * D * 2 : nq * NG * 2;
  const uint32_t vmeta = nq * NG * 2;
  const bool zero_planes = FMT != KVQ_FMT_SYMMETRIC;
  uint32_t total = 2 * code_bytes + kmeta + vmeta;
  if (zero_planes) total += kmeta + vmeta;
  mbar_expect_tx(&bars[stage], total);
  // a chunk is one 64-token page of a paged cache: tok_ptr finds its rows
  bulk_g2s(st + C::KC_OFF, tok_ptr<uint8_t>(g, KVQ_PLANE_K_CODES, b, hkv, c0), code_bytes,
           &bars[stage]);
  bulk_g2s(st + C::VC_OFF, tok_ptr<uint8_t>(g, KVQ_PLANE_V_CODES, b, hkv, c0), code_bytes,
           &bars[stage]);
  if (FMT == KVQ_FMT_KIVI) {
    bulk_g2s(st + C::KS_OFF, blk_ptr<__half>(g, KVQ_PLANE_K_SCALE, b, hkv, c0 / 32), kmeta,
             &bars[stage]);
    bulk_g2s(st + C::KZ_OFF, blk_ptr<__half>(g, KVQ_PLANE_K_ZERO, b, hkv, c0 / 32), kmeta,
             &bars[stage]);
  } else {
    bulk_g2s(st + C::KS_OFF, tok_ptr<__half>(g, KVQ_PLANE_K_SCALE, b, hkv, c0), kmeta,
             &bars[stage]);
    if (zero_planes)
      bulk_g2s(st + C::KZ_OFF, tok_ptr<__half>(g, KVQ_PLANE_K_ZERO, b, hkv, c0), kmeta,
               &bars[stage]);
  }
  bulk_g2s(st + C::VS_OFF, tok_ptr<__half>(g, KVQ_PLANE_V_SCALE, b, hkv, c0), vmeta,
           &bars[stage]);
  if (zero_planes)
    bulk_g2s(st + C::VZ_OFF, tok_ptr<__half>(g, KVQ_PLANE_V_ZERO, b, hkv, c0), vmeta,
             &bars[stage]);
}

// Initialise the stage barriers and issue the first STAGES chunks of a split,
// lane c of warp 0 the copies of chunk c (the chunks' copies are issued
// together rather than one chunk after another).  Every thread of the CTA
// calls it.
template <int D, int BITS, int FMT, int STAGES>
__device__ void split_prologue(const Geom& g, int b, int hkv, const SplitPlan& sp,
                               unsigned char* smem, uint64_t* bars) {
  static_assert(STAGES <= 32, "one lane per stage");
  if (threadIdx.x < 32) {
    if (threadIdx.x == 0) {
      for (int i = 0; i < STAGES; ++i) mbar_init(&bars[i], 1);
      asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncwarp();
    if ((int)threadIdx.x < min(STAGES, sp.nchunks))
      split_issue<D, BITS, FMT, STAGES>(g, b, hkv, sp, threadIdx.x, smem, bars);
  }
  __syncthreads();
}

// Merge the tagged split partials of the query heads of kv head hkv of
// sequence b into out, polling each word until it carries `tag`.  Each
// output pair takes m, l and its two values from every split in one pass.
template <int D>
__device__ void merge_tagged(const Geom& g, __nv_bfloat16* __restrict__ out, int b, int hkv,
                             int grp, int S, int sstride, uint32_t tag, int* err) {
  const uint64_t* wbase = reinterpret_cast<const uint64_t*>(g.pl[KVQ_PLANE_WORKSPACE].p) +
                          ((int64_t)b * g.Hq + hkv * grp) * sstride * (D + kWsStride);
  constexpr int SB = 16;
  for (int i = threadIdx.x; i < grp * (D / 2); i += blockDim.x) {
    const int row = i / (D / 2), d = 2 * (i % (D / 2));
    const uint64_t* w = wbase + (int64_t)row * sstride * (D + kWsStride);
    float M = -INFINITY, L = 0.f, a0 = 0.f, a1 = 0.f;
    for (int s0 = 0; s0 < S; s0 += SB) {
      float ms[SB], ls[SB], v0[SB], v1[SB];
      // every word of the block is loaded before any is checked (the loads
      // are in flight together: one L2 round trip per poll)
      uint64_t wv[SB][4];
      for (long it = 0;; ++it) {
#pragma unroll
        for (int k = 0; k < SB; ++k) {
          const uint64_t* ws = w + min(s0 + k, S - 1) * (D + kWsStride);
          ld_tagged2(ws, wv[k][0], wv[k][1]);        // rows of D + 2 words, d even:
          ld_tagged2(ws + 2 + d, wv[k][2], wv[k][3]); // both pairs 16-byte aligned
        }
        bool ok = true;
#pragma unroll
        for (int k = 0; k < SB; ++k)
          if (s0 + k < S)
#pragma unroll
            for (int c = 0; c < 4; ++c) ok = ok && tag_is(wv[k][c], tag);
        if (ok) break;
        if (it > kPollLimit) {
          atomicOr(err, 2);
          break;
        }
      }
#pragma unroll
      for (int k = 0; k < SB; ++k) {
        const bool live = s0 + k < S;
        ms[k] = live ? tagged_value(wv[k][0]) : -INFINITY;
        ls[k] = live ? tagged_value(wv[k][1]) : 0.f;
        v0[k] = live ? tagged_value(wv[k][2]) : 0.f;
        v1[k] = live ? tagged_value(wv[k][3]) : 0.f;
      }
      float Mb = M;
#pragma unroll
      for (int k = 0; k < SB; ++k) Mb = fmaxf(Mb, ms[k]);
      if (Mb == -INFINITY) continue;
      const float r = M == -INFINITY ? 0.f : expf(M - Mb);
      L *= r;
      a0 *= r;
      a1 *= r;
#pragma unroll
      for (int k = 0; k < SB; ++k) {
        const float f = ms[k] == -INFINITY ? 0.f : expf(ms[k] - Mb);
        L += f * ls[k];
        a0 += f * v0[k];
        a1 += f * v1[k];
      }
      M = Mb;
    }
    const float inv = L > 0.f ? 1.f / L : 0.f;
    *reinterpret_cast<__nv_bfloat162*>(out + ((int64_t)b * g.Hq + hkv * grp + row) * D + d) =
        __floats2bfloat162_rn(a0 * inv, a1 * inv);
  }
}

// One split of one (sequence, kv head): blockIdx-independent, so a fused
// kernel can run several per CTA.  T = tokens stored (read by the caller);
// `splits` splits share the tokens.  qg: the query rows of the kv head's
// query heads (row hl at qg + hl D, global or shared memory).  The CTA has
// NW warps (a multiple of 4): each step takes NW / 4 chunks, one 16-token
// tile per warp.  smem: at least attn_smem_bytes<D, BITS, FMT, STAGES, NW>()
// bytes; full_bar: STAGES mbarriers in shared memory.  With `prologue_done`
// the caller already ran split_prologue (to start the copies early).  The
// split partials of query head (b, h) sit in the workspace at element
// ((b Hq + h) sstride + split) (D + 2) (sstride >= splits).  With tag == 0
// they are floats and the last split CTA to arrive (an atomic counter)
// merges; otherwise they are tagged words and the CTA called with `merger`
// polls the other splits' words and merges.
template <int D, int BITS, int FMT, int STAGES, int NW>
__device__ void decode_split(const Geom& g, const __nv_bfloat16* qg, float scale, int* err,
                             __nv_bfloat16* __restrict__ out, int split, int splits, int sstride,
                             int hkv, int b, int T, unsigned char* smem, uint64_t* full_bar,
                             bool prologue_done, uint32_t tag = 0, bool merger = false) {
  using C = Cfg<D, BITS, FMT>;
  constexpr int NG = C::NG, KSTEP = C::KSTEP, NT_PV = C::NT_PV;
  constexpr int GCH = NW / kWarps;                    // chunks per step
  static_assert(NW % kWarps == 0 && STAGES >= GCH, "warps cover whole chunks");
  __shared__ float red_m[NW][16], red_l[NW][16], wsc[NW][16];
  __shared__ int last_cta;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gid = lane >> 2, tid = lane & 3;
  const SplitPlan sp = split_plan<FMT>(g, T, splits, split);
  const int ts = sp.ts, te = sp.te, tq = sp.tq;
  const int grp = g.Hq / g.H;
  const float l2e = 1.4426950408889634f;
  const float qk_scale = scale * l2e;                 // scores in log2 units

  // ---- query fragments (rows = heads gid, gid + 8) and per-group sums -----
  uint32_t qa[KSTEP][4];
  float qsum[NG][2];
  float qv[2][NG][8];                                 // this thread's 8 channels per group
  for (int r = 0; r < 2; ++r) {
    const int hl = gid + 8 * r;
    for (int gq = 0; gq < NG; ++gq) {
      uint4 u = make_uint4(0, 0, 0, 0);
      if (hl < grp) u = *reinterpret_cast<const uint4*>(qg + hl * D + 32 * gq + 8 * tid);
      const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&u);
      float s = 0.f;
      for (int e = 0; e < 4; ++e) {
        const float2 f = __bfloat1622float2(h2[e]);
        qv[r][gq][2 * e] = f.x;
        qv[r][gq][2 * e + 1] = f.y;
        s += f.x;
        s += f.y;
      }
      qsum[gq][r] = s;       // partial over this thread's 8 channels
    }
  }
  for (int gq = 0; gq < NG; ++gq)
    for (int r = 0; r < 2; ++r) {
      qsum[gq][r] += __shfl_xor_sync(0xffffffffu, qsum[gq][r], 1);
      qsum[gq][r] += __shfl_xor_sync(0xffffffffu, qsum[gq][r], 2);
    }
  // dst = bf16(q * mul); lo (if given) = bf16 of the remainder, so that
  // hi + lo carries about 16 significant bits of q * mul
  auto build_q = [&](uint32_t (&dst)[KSTEP][4], const float (*mul)[8], uint32_t (*lo)[4]) {
    // mul[gq][e]: per-channel factor of this thread's channels (KIVI block
    // scales), or nullptr
    for (int gq = 0; gq < NG; ++gq)
      for (int s = 0; s < 2; ++s) {
        const int ks = 2 * gq + s;
        for (int half = 0; half < 2; ++half)
          for (int r = 0; r < 2; ++r) {
            const int e0 = qk_chan<BITS>(s, half, 0), e1 = qk_chan<BITS>(s, half, 1);
            float v0 = qv[r][gq][e0], v1 = qv[r][gq][e1];
            if (mul) {
              v0 *= mul[gq][e0];
              v1 *= mul[gq][e1];
            }
            const __nv_bfloat162 hb = __floats2bfloat162_rn(v0, v1);
            dst[ks][half * 2 + r] = *reinterpret_cast<const uint32_t*>(&hb);
            if (lo) {
              const float2 hf = __bfloat1622float2(hb);
              lo[ks][half * 2 + r] = pack_bf16(v0 - hf.x, v1 - hf.y);
            }
          }
      }
  };
  build_q(qa, nullptr, nullptr);

  // ---- running softmax state and accumulators -----------------------------
  float m_run[2] = {-INFINITY, -INFINITY}, l_run[2] = {0.f, 0.f};
  float o[NT_PV][4];
  for (int j = 0; j < NT_PV; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
  float cterm[2][NG];
  for (int gq = 0; gq < NG; ++gq) cterm[0][gq] = cterm[1][gq] = 0.f;

  // ---- chunk pipeline ------------------------------------------------------
  const int nchunks = sp.nchunks;
  const bool leader = threadIdx.x == 0;
  if (!prologue_done) split_prologue<D, BITS, FMT, STAGES>(g, b, hkv, sp, smem, full_bar);

  bool timed_out = false;
  const uint32_t kmask = BITS == 4 ? 0x000F000Fu : 0x00030003u;
  const int zbias = FMT == KVQ_FMT_SYMMETRIC ? (1 << (BITS - 1)) : 0;

  const int wchunk = warp / kWarps;                  // chunk of the step this warp takes
  const int tile_off = 16 * (warp % kWarps);         // its tile's row offset in the chunk
  int chunk = 0;
  for (; chunk < nchunks; chunk += GCH) {
    const int my = chunk + wchunk;
    bool ok = true;
    if (my < nchunks) ok = mbar_wait(&full_bar[my % STAGES], (my / STAGES) & 1);
    if (__syncthreads_or(!ok)) {        // the same decision in every thread
      timed_out = true;
      break;
    }
    const unsigned char* st = smem + (my % STAGES) * C::STAGE_B;
    const int t0 = ts + my * kCT + tile_off;         // this warp's tile
    if (my < nchunks && t0 < te) {
      // every token of an affine/symmetric cache is coded; KIVI keeps the
      // newest tokens in full precision
      const bool coded = FMT != KVQ_FMT_KIVI || t0 < tq;
      float sacc[2][4];                              // S for n-tiles 0, 1 (tokens t0 + 8nt + col)
      // ---------------- scores ----------------
      if (coded && FMT != KVQ_FMT_KIVI) {
        float acc[NG][2][4];
        for (int gq = 0; gq < NG; ++gq)
          for (int nt = 0; nt < 2; ++nt) acc[gq][nt][0] = acc[gq][nt][1] = acc[gq][nt][2] = acc[gq][nt][3] = 0.f;
        for (int nt = 0; nt < 2; ++nt) {
          const unsigned char* row = st + C::KC_OFF + (tile_off + 8 * nt + gid) * C::CODE_B;
          for (int gq = 0; gq < NG; ++gq) {
            uint32_t w;
            if (BITS == 4) w = *reinterpret_cast<const uint32_t*>(row + 16 * gq + 4 * tid);
            else {
              const uint32_t v = *reinterpret_cast<const uint16_t*>(row + 8 * gq + 2 * tid);
              w = v | (v << 14);
            }
            for (int s = 0; s < 2; ++s) {
              const uint32_t b0 = magic2(w >> (BITS == 4 ? 8 * s : 8 * s), kmask);
              const uint32_t b1 = magic2(w >> (BITS == 4 ? 8 * s + 4 : 8 * s + 4), kmask);
              mma16816(acc[gq][nt], qa[2 * gq + s], b0, b1);
            }
          }
        }
        // apply per-token scale and offset: columns 2tid, 2tid+1 of each n-tile
        const __half* ksc = reinterpret_cast<const __half*>(st + C::KS_OFF);
        const __half* kze = reinterpret_cast<const __half*>(st + C::KZ_OFF);
        for (int nt = 0; nt < 2; ++nt)
          for (int cc = 0; cc < 2; ++cc) {
            const int rr = tile_off + 8 * nt + 2 * tid + cc;     // row within chunk
            float s0 = 0.f, s1 = 0.f;
            for (int gq = 0; gq < NG; ++gq) {
              const float sc = __half2float(ksc[rr * NG + gq]);
              const float mz = FMT == KVQ_FMT_SYMMETRIC ? -(float)zbias * sc
                                                       : __half2float(kze[rr * NG + gq]);
              const float off = mz - 128.f * sc;
              s0 += sc * acc[gq][nt][cc] + off * qsum[gq][0];
              s1 += sc * acc[gq][nt][2 + cc] + off * qsum[gq][1];
            }
            sacc[nt][cc] = s0;
            sacc[nt][2 + cc] = s1;
          }
      } else if (coded) {  // KIVI: per-channel block scale folded into q
        const int blk_row = (tile_off) / 32;            // block within the chunk
        const __half* ksc = reinterpret_cast<const __half*>(st + C::KS_OFF) + blk_row * D;
        const __half* kze = reinterpret_cast<const __half*>(st + C::KZ_OFF) + blk_row * D;
        float mul[NG][8];
        for (int gq = 0; gq < NG; ++gq)
          for (int e = 0; e < 8; ++e) mul[gq][e] = __half2float(ksc[32 * gq + 8 * tid + e]);
        uint32_t qk[KSTEP][4], ql[KSTEP][4];
        build_q(qk, mul, ql);
        // constant: sum_d q_d m_d - 128 sum_d q'_d, q' = hi + lo as fed to the MMAs
        float cst[2] = {0.f, 0.f};
        for (int gq = 0; gq < NG; ++gq)
          for (int e = 0; e < 8; ++e) {
            const float mz = __half2float(kze[32 * gq + 8 * tid + e]);
            for (int r = 0; r < 2; ++r) {
              const float qr = qv[r][gq][e];
              const float qx = qr * mul[gq][e];
              const float qh = __bfloat162float(__float2bfloat16_rn(qx));
              const float ql2 = __bfloat162float(__float2bfloat16_rn(qx - qh));
              cst[r] += qr * mz - 128.f * (qh + ql2);
            }
          }
        for (int r = 0; r < 2; ++r) {
          cst[r] += __shfl_xor_sync(0xffffffffu, cst[r], 1);
          cst[r] += __shfl_xor_sync(0xffffffffu, cst[r], 2);
        }
        for (int nt = 0; nt < 2; ++nt) {
          float acc[4] = {0.f, 0.f, 0.f, 0.f};
          const unsigned char* row = st + C::KC_OFF + (tile_off + 8 * nt + gid) * C::CODE_B;
          for (int gq = 0; gq < NG; ++gq) {
            uint32_t w;
            if (BITS == 4) w = *reinterpret_cast<const uint32_t*>(row + 16 * gq + 4 * tid);
            else {
              const uint32_t v = *reinterpret_cast<const uint16_t*>(row + 8 * gq + 2 * tid);
              w = v | (v << 14);
            }
            for (int s = 0; s < 2; ++s) {
              const uint32_t b0 = magic2(w >> (8 * s), kmask), b1 = magic2(w >> (8 * s + 4), kmask);
              mma16816(acc, qk[2 * gq + s], b0, b1);
              mma16816(acc, ql[2 * gq + s], b0, b1);
            }
          }
          sacc[nt][0] = acc[0] + cst[0];
          sacc[nt][1] = acc[1] + cst[0];
          sacc[nt][2] = acc[2] + cst[1];
          sacc[nt][3] = acc[3] + cst[1];
        }
      } else {  // full-precision tokens (KIVI residual ring)
        for (int nt = 0; nt < 2; ++nt) {
          float acc[4] = {0.f, 0.f, 0.f, 0.f};
          const int t = t0 + 8 * nt + gid;
          const bool ok = t < te;
          const int slot = t % g.ring;
          const __nv_bfloat16* krow =
              plane_ptr<__nv_bfloat16>(g, KVQ_PLANE_K_FULL, b, hkv, ok ? slot : 0);
          for (int gq = 0; gq < NG; ++gq) {
            uint4 u = ok ? *reinterpret_cast<const uint4*>(krow + 32 * gq + 8 * tid)
                         : make_uint4(0, 0, 0, 0);
            const uint16_t* e = reinterpret_cast<const uint16_t*>(&u);
            for (int s = 0; s < 2; ++s) {
              const uint32_t b0 = pack_raw(e[qk_chan<BITS>(s, 0, 0)], e[qk_chan<BITS>(s, 0, 1)]);
              const uint32_t b1 = pack_raw(e[qk_chan<BITS>(s, 1, 0)], e[qk_chan<BITS>(s, 1, 1)]);
              mma16816(acc, qa[2 * gq + s], b0, b1);
            }
          }
          for (int i = 0; i < 4; ++i) sacc[nt][i] = acc[i];
        }
      }
      // ---------------- online softmax (log2 domain) ----------------
      float mx[2] = {-INFINITY, -INFINITY};
      for (int nt = 0; nt < 2; ++nt)
        for (int cc = 0; cc < 2; ++cc) {
          const int t = t0 + 8 * nt + 2 * tid + cc;
          for (int r = 0; r < 2; ++r) {
            float v = sacc[nt][2 * r + cc] * qk_scale;
            if (t >= te) v = -INFINITY;
            sacc[nt][2 * r + cc] = v;
            mx[r] = fmaxf(mx[r], v);
          }
        }
      float alpha[2];
      for (int r = 0; r < 2; ++r) {
        mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 1));
        mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 2));
        const float mn = fmaxf(m_run[r], mx[r]);
        alpha[r] = mn == -INFINITY ? 1.f : exp2f(m_run[r] - mn);
        m_run[r] = mn;
        l_run[r] *= alpha[r];
      }
      for (int j = 0; j < NT_PV; ++j) {
        o[j][0] *= alpha[0]; o[j][1] *= alpha[0];
        o[j][2] *= alpha[1]; o[j][3] *= alpha[1];
      }
      for (int gq = 0; gq < NG; ++gq) {
        cterm[0][gq] *= alpha[0];
        cterm[1][gq] *= alpha[1];
      }
      float p[2][4];
      for (int nt = 0; nt < 2; ++nt)
        for (int i = 0; i < 4; ++i) {
          const int r = i >> 1;
          const float v = sacc[nt][i];
          p[nt][i] = v == -INFINITY ? 0.f : exp2f(v - m_run[r]);
          l_run[r] += p[nt][i];
        }
      // ---------------- P V ----------------
      // A fragment: a0 = (row gid, tokens 2tid, 2tid+1) = p[0][0..1], a1 = row
      // gid+8 = p[0][2..3], a2 = tokens 2tid+8, +9 = p[1][0..1], a3 = p[1][2..3].
      const int tok[4] = {2 * tid, 2 * tid + 1, 2 * tid + 8, 2 * tid + 9};
      if (coded) {
        const __half* vsc = reinterpret_cast<const __half*>(st + C::VS_OFF);
        const __half* vze = reinterpret_cast<const __half*>(st + C::VZ_OFF);
        for (int gv = 0; gv < NG; ++gv) {
          float sv[4], mz[4];
          for (int i = 0; i < 4; ++i) {
            const int rr = tile_off + tok[i];
            const bool ok = t0 + tok[i] < te;
            const float sc = ok ? __half2float(vsc[rr * NG + gv]) : 0.f;
            sv[i] = sc;
            mz[i] = !ok ? 0.f
                : FMT == KVQ_FMT_SYMMETRIC ? -(float)zbias * sc : __half2float(vze[rr * NG + gv]);
          }
          // p is indexed [nt][2r + cc]; token tok[i]: nt = i >> 1, cc = i & 1.
          // The fp16 MMA sees fp16(p s) (c + 1024); the offset term removes
          // exactly 1024 fp16(p s) and adds p m.
          float ps[2][4];
          for (int nt = 0; nt < 2; ++nt)
            for (int i = 0; i < 4; ++i)
              ps[nt][i] = __half2float(__float2half_rn(p[nt][i] * sv[2 * nt + (i & 1)]));
          uint32_t a[4];
          a[0] = pack_f16(ps[0][0], ps[0][1]);
          a[1] = pack_f16(ps[0][2], ps[0][3]);
          a[2] = pack_f16(ps[1][0], ps[1][1]);
          a[3] = pack_f16(ps[1][2], ps[1][3]);
          for (int r = 0; r < 2; ++r)
            for (int nt = 0; nt < 2; ++nt)
              for (int cc = 0; cc < 2; ++cc)
                cterm[r][gv] += p[nt][2 * r + cc] * mz[2 * nt + cc] - 1024.f * ps[nt][2 * r + cc];
          // B: codes of tokens (2tid, 2tid+1) and (2tid+8, 2tid+9) at channels
          // 32 gv + 4 gid + jj, jj = 0..3 (one n-tile per jj)
          uint32_t cw[4];
          for (int i = 0; i < 4; ++i) {
            const unsigned char* row = st + C::VC_OFF + (tile_off + tok[i]) * C::CODE_B;
            cw[i] = BITS == 4 ? *reinterpret_cast<const uint16_t*>(row + 16 * gv + 2 * gid)
                              : *reinterpret_cast<const uint8_t*>(row + 8 * gv + gid);
          }
          const uint32_t x01 = cw[0] | (cw[1] << 16), x23 = cw[2] | (cw[3] << 16);
          for (int jj = 0; jj < 4; ++jj)
            mma16816_f16(o[4 * gv + jj], a, magic2h(x01 >> (BITS * jj), kmask),
                         magic2h(x23 >> (BITS * jj), kmask));
        }
      } else {  // full-precision values (bf16 -> fp16 for the fp16 MMA)
        uint32_t a[4];
        a[0] = pack_f16(p[0][0], p[0][1]);
        a[1] = pack_f16(p[0][2], p[0][3]);
        a[2] = pack_f16(p[1][0], p[1][1]);
        a[3] = pack_f16(p[1][2], p[1][3]);
        for (int gv = 0; gv < NG; ++gv) {
          uint2 vw[4];
          for (int i = 0; i < 4; ++i) {
            const int t = t0 + tok[i];
            const bool ok = t < te;
            const __nv_bfloat16* vrow =
                plane_ptr<__nv_bfloat16>(g, KVQ_PLANE_V_FULL, b, hkv, ok ? t % g.ring : 0);
            vw[i] = ok ? *reinterpret_cast<const uint2*>(vrow + 32 * gv + 4 * gid)
                       : make_uint2(0, 0);
          }
          for (int jj = 0; jj < 4; ++jj) {
            auto el = [&](int i) {
              const __nv_bfloat16* e = reinterpret_cast<const __nv_bfloat16*>(&vw[i]);
              return __bfloat162float(e[jj]);
            };
            mma16816_f16(o[4 * gv + jj], a, pack_f16(el(0), el(1)), pack_f16(el(2), el(3)));
          }
        }
      }
    }
    __syncthreads();                                  // every warp is done with the stages
    if (leader && chunk + STAGES < nchunks) {
      // shared: the stages were read by generic loads; global: in the fused
      // step a chunk may hold rows stored earlier in the same kernel
      asm volatile("fence.proxy.async;" ::: "memory");
      for (int j = 0; j < GCH && chunk + j + STAGES < nchunks; ++j)
        split_issue<D, BITS, FMT, STAGES>(g, b, hkv, sp, chunk + j + STAGES, smem, full_bar);
    }
  }
  if (timed_out) {
    // flag the error, then drain (again bounded) the copies still in flight
    if (threadIdx.x == 0) {
      atomicOr(err, 1);
      for (int c = chunk; c < min(nchunks, chunk + STAGES); ++c)
        mbar_wait(&full_bar[c % STAGES], (c / STAGES) & 1);
    }
    __syncthreads();
    if (threadIdx.x == 0)
      for (int i = 0; i < STAGES; ++i) mbar_inval(&full_bar[i]);
    __syncthreads();
    return;
  }
  // ---- finish: reduce l and the offset terms over the 4 lanes of a row ----
  for (int r = 0; r < 2; ++r) {
    l_run[r] += __shfl_xor_sync(0xffffffffu, l_run[r], 1);
    l_run[r] += __shfl_xor_sync(0xffffffffu, l_run[r], 2);
    for (int gv = 0; gv < NG; ++gv) {
      cterm[r][gv] += __shfl_xor_sync(0xffffffffu, cterm[r][gv], 1);
      cterm[r][gv] += __shfl_xor_sync(0xffffffffu, cterm[r][gv], 2);
    }
  }
  // o columns: n-tile j = 4 gv + jj holds channels 32 gv + 4 col + jj at
  // columns col = 2tid, 2tid + 1
  constexpr int OS = D + 1;                           // odd row stride: no bank conflicts
  float* osm = reinterpret_cast<float*>(smem);        // [NW][16][OS]
  __syncthreads();
  for (int j = 0; j < NT_PV; ++j) {
    const int gv = j >> 2, jj = j & 3;
    for (int i = 0; i < 4; ++i) {
      const int row = gid + 8 * (i >> 1), col = 2 * tid + (i & 1);
      const int d = 32 * gv + 4 * col + jj;
      osm[(warp * 16 + row) * OS + d] = o[j][i] + cterm[i >> 1][gv];
    }
  }
  if (tid == 0) {
    red_m[warp][gid] = m_run[0];
    red_m[warp][gid + 8] = m_run[1];
    red_l[warp][gid] = l_run[0];
    red_l[warp][gid + 8] = l_run[1];
  }
  __syncthreads();
  // per row: the warps' weights exp2(m_w - M), M = max_w m_w (0 for empty warps)
  if (threadIdx.x < 16) {
    const int row = threadIdx.x;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < NW; ++w) M = fmaxf(M, red_m[w][row]);
#pragma unroll
    for (int w = 0; w < NW; ++w)
      wsc[w][row] = red_m[w][row] == -INFINITY ? 0.f : exp2f(red_m[w][row] - M);
  }
  __syncthreads();
  // merge the warps and write the split's partial (m in natural-log units)
  for (int i = threadIdx.x; i < grp * (D + kWsStride); i += blockDim.x) {
    const int row = i / (D + kWsStride), c = i % (D + kWsStride);
    float val = 0.f;
    if (c == 0) {
      float M = -INFINITY;
#pragma unroll
      for (int w = 0; w < NW; ++w) M = fmaxf(M, red_m[w][row]);
      val = M == -INFINITY ? -INFINITY : M / l2e;
    } else if (c == 1) {
#pragma unroll
      for (int w = 0; w < NW; ++w) val += wsc[w][row] * red_l[w][row];
    } else {
#pragma unroll
      for (int w = 0; w < NW; ++w) val += wsc[w][row] * osm[(w * 16 + row) * OS + c - 2];
    }
    const int64_t wi = (((int64_t)b * g.Hq + hkv * grp + row) * sstride + split) * (D + kWsStride) + c;
    if (tag) st_tagged(reinterpret_cast<uint64_t*>(g.pl[KVQ_PLANE_WORKSPACE].p) + wi, val, tag);
    else reinterpret_cast<float*>(g.pl[KVQ_PLANE_WORKSPACE].p)[wi] = val;
  }
  if (tag) {
    // tagged partials: the merger polls them; everyone else is done
    __syncthreads();
    if (threadIdx.x == 0)
      for (int i = 0; i < STAGES; ++i) mbar_inval(&full_bar[i]);
    if (merger) merge_tagged<D>(g, out, b, hkv, grp, splits, sstride, tag, err);
    __syncthreads();
    return;
  }
  // ---- the last split CTA of this (sequence, kv head) merges all splits ----
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    const unsigned prev = atomicAdd(&g.counters[b * g.H + hkv], 1u);
    last_cta = prev == (unsigned)splits - 1;
  }
  __syncthreads();
  if (threadIdx.x == 0)                       // all copies were consumed: retire the barriers
    for (int i = 0; i < STAGES; ++i) mbar_inval(&full_bar[i]);
  if (!last_cta) {
    __syncthreads();
    return;
  }
  __threadfence();
  const float* wbase = reinterpret_cast<const float*>(g.pl[KVQ_PLANE_WORKSPACE].p) +
                       ((int64_t)b * g.Hq + hkv * grp) * sstride * (D + kWsStride);
  // each output pair loads the m, l and values of all splits of its row in
  // one pass (blocks of 16 splits, rescaled online), then normalises
  const int S = splits;
  constexpr int SB = 16;
  for (int i = threadIdx.x; i < grp * (D / 2); i += blockDim.x) {
    const int row = i / (D / 2), d = 2 * (i % (D / 2));
    const float* w = wbase + (int64_t)row * sstride * (D + kWsStride);
    float M = -INFINITY, L = 0.f, a0 = 0.f, a1 = 0.f;
    for (int s0 = 0; s0 < S; s0 += SB) {
      float ms[SB], ls[SB];
      float2 v[SB];
#pragma unroll
      for (int k = 0; k < SB; ++k) {
        const int sp = s0 + k;
        const float* ws = w + sp * (D + kWsStride);
        ms[k] = sp < S ? __ldcg(ws) : -INFINITY;
        ls[k] = sp < S ? __ldcg(ws + 1) : 0.f;
        v[k] = sp < S ? __ldcg(reinterpret_cast<const float2*>(ws + 2 + d)) : make_float2(0.f, 0.f);
      }
      float Mb = M;
#pragma unroll
      for (int k = 0; k < SB; ++k) Mb = fmaxf(Mb, ms[k]);
      if (Mb == -INFINITY) continue;
      const float r = M == -INFINITY ? 0.f : expf(M - Mb);
      L *= r;
      a0 *= r;
      a1 *= r;
#pragma unroll
      for (int k = 0; k < SB; ++k) {
        const float f = ms[k] == -INFINITY ? 0.f : expf(ms[k] - Mb);
        L += f * ls[k];
        a0 += f * v[k].x;
        a1 += f * v[k].y;
      }
      M = Mb;
    }
    const float inv = L > 0.f ? 1.f / L : 0.f;
    *reinterpret_cast<__nv_bfloat162*>(out + ((int64_t)b * g.Hq + hkv * grp + row) * D + d) =
        __floats2bfloat162_rn(a0 * inv, a1 * inv);
  }
  if (threadIdx.x == 0) g.counters[b * g.H + hkv] = 0;   // ready for the next call
  __syncthreads();
}

template <int D, int BITS, int FMT, int STAGES = kStages, int NW = kWarps>
__host__ __device__ constexpr size_t attn_smem_bytes() {
  using C = Cfg<D, BITS, FMT>;
  return (size_t)STAGES * C::STAGE_B > (size_t)NW * 16 * (D + 1) * sizeof(float)
             ? (size_t)STAGES * C::STAGE_B : (size_t)NW * 16 * (D + 1) * sizeof(float);
}


}  // namespace dattn
}  // namespace kvq
