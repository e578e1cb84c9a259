// Causal GQA prefill attention over the stored reconstruction on the
// 5th-generation tensor cores (tcgen05), Sections 3.1-3.3: the L newest
// queries attend to every token up to their own position, and every key and
// value is the cache's reconstruction (codes x scale + offset, or the
// full-precision residual window of a KIVI cache).
//
// One CTA = 256 query rows of one (sequence, kv head): the g query heads of
// the kv head x 256/g consecutive queries, head-major, split into two
// 128-row query tiles A (rows 0..127) and B (rows 128..255) that share every
// reconstructed key/value tile.  Keys and values stream in tiles of 64
// tokens.  Four roles:
//   producers (warps 8-11): reconstruct each K/V tile once for both query
//     tiles: K as a bf16 high part (the fp32 value truncated) plus the bf16
//     of the remainder (about 16 significant bits: large logits need more
//     than bf16's 8), V as fp16 computed in packed half2 arithmetic
//     (code x scale + offset, one rounding), into double-buffered shared
//     tiles in the 128-byte-swizzled K-major layout of the MMA descriptors
//     (V transposed: D rows, tokens along K);
//   issuer (warp 12, one thread): per KV tile j, first O_X += P_X V of tile
//     j - 1 into a TMEM accumulator (128 x D fp32) per query tile X = A, B
//     (this frees tile j - 1's K/V buffer, so the producers run a tile
//     ahead), then S_X = Q_X K_hi^T + Q_X K_lo^T of tile j into
//     double-buffered TMEM tiles (128 x 64 fp32); completions are signalled
//     by tcgen05.commit on mbarriers;
//   softmax A (warps 0-3) and B (warps 4-7): thread r owns row r of its
//     query tile (TMEM lane r): reads the 64 scores, masks causally, keeps
//     the running maximum m and sum l in log2 units, writes P as fp16 into
//     its query tile's P buffer.  O is rescaled (in TMEM) only when a row's
//     maximum grows by more than 8 (so P stays <= 2^8 in fp16); the final
//     O / l is stored as bf16.
// Every wait is bounded and also gives up when another role has timed out;
// the issuer drains its MMAs before TMEM is freed, and a timed-out CTA
// stores nothing and sets the library's error word.
#include <math.h>

#include "tc_common.cuh"

namespace kvq {
namespace {
using namespace tc;

constexpr int kM = 128;              // rows per query tile (MMA M)
constexpr int kTok = 64;             // tokens per KV tile
constexpr int kRowsCta = 2 * kM;     // query rows per CTA
constexpr int kThreads = 14 * 32;    // 8 softmax, 4 producer, 1 issuer, 1 loader warp
constexpr int kKvBufs = 2;           // reconstructed K/V tile buffers
constexpr int kRaw = 3;              // packed-tile stages (bulk copies run up to 3 tiles ahead)
constexpr float kRescale = 8.f;      // log2 growth of a row maximum that forces a rescale

// Shared memory (bytes from a 1024-aligned base).
template <int D, int BITS>
struct M256Layout {
  static constexpr int QT = kM * D * 2;             // one query tile: D/64 atoms of 16 KB
  static constexpr int Q_OFF = 0;
  static constexpr int KV_OFF = 2 * QT;
  static constexpr int KH = 0;                      // K hi: D/64 atoms of 64 rows x 128 B
  static constexpr int KL = kTok * D * 2;           // K lo: the same
  static constexpr int VT = 2 * kTok * D * 2;       // V^T: D rows x 128 B (64 tokens)
  static constexpr int KV_B = VT + D * 128;
  // packed tile as stored in the cache planes: 64 code rows of K and of V,
  // then four metadata pieces of 4 D bytes each (per-token group scales and
  // offsets of 64 tokens, or KIVI's per-channel scales and offsets of the
  // tile's two 32-token key blocks)
  static constexpr int CROW = D * BITS / 8;         // code bytes per token
  static constexpr int RKC = 0, RVC = kTok * CROW;
  static constexpr int RKS = 2 * kTok * CROW, RKZ = RKS + 4 * D, RVS = RKZ + 4 * D,
                       RVZ = RVS + 4 * D;
  static constexpr int RAW_B = RVZ + 4 * D;
  static constexpr int RAW_OFF = KV_OFF + kKvBufs * KV_B;
  static constexpr int TOTAL = RAW_OFF + kRaw * RAW_B;
  static constexpr int ALLOC = TOTAL + 1024;        // alignment slack
};

// Byte offset of 16-byte chunk c of row r in a K-major 128-byte-swizzled
// tile (rows of 128 bytes, 8-row groups 1024 bytes apart).
__device__ __forceinline__ int sw128(int r, int c) {
  return (r >> 3) * 1024 + (r & 7) * 128 + ((c ^ (r & 7)) << 4);
}

__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}
// Packed fp32 pairs (two lanes of one 64-bit register).
__device__ __forceinline__ uint64_t f2pack(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void f2unpack(uint64_t v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ uint64_t ffma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t fadd2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}

__device__ __forceinline__ uint32_t pack_h2(float lo, float hi) {
  __half2 v = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t r[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,"
      "%13,%14,%15,%16};\n"
      ::"r"(taddr), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]),
        "r"(r[6]), "r"(r[7]), "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]),
        "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}
__device__ __forceinline__ void tmem_wait_st() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// D (+)= A B with A (M x 16, 16-bit elements packed two per 32-bit column)
// read from tensor memory and B from shared memory.
__device__ __forceinline__ void umma_ts(uint32_t tmem_d, uint32_t tmem_a, uint64_t bdesc,
                                        uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}\n"
      ::"r"(tmem_d), "r"(tmem_a), "l"(bdesc), "r"(idesc), "r"(accumulate));
}

// True in exactly one lane of the (fully active) warp.
__device__ __forceinline__ bool elect_one() {
  uint32_t p;
  asm volatile(
      "{\n .reg .pred e;\n elect.sync _|e, 0xffffffff;\n selp.u32 %0, 1, 0, e;\n}\n"
      : "=r"(p));
  return p != 0;
}

// Non-blocking probe of an mbarrier phase.
__device__ __forceinline__ bool mbar_test(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok) : "r"(smem_u32(bar)), "r"(parity) : "memory");
  return ok != 0;
}

__device__ __forceinline__ void bulk_copy(void* dst, const void* src, uint32_t bytes,
                                          uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
      ::"r"(smem_u32(dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar)) : "memory");
}

// Bounded mbarrier wait whose result is the same in every lane of the warp
// (the warp-collective TMEM loads and stores that follow need all lanes).
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort) {
  const bool w = mbar_wait_or_abort(bar, parity, abort);
  return __all_sync(0xffffffffu, w);
}

// Barrier of the four producer warps (named barrier 1) that also returns
// whether `ok` held in every producer thread, so all of them leave the tile
// loop together.
__device__ __forceinline__ bool producers_all(bool ok) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n"
      " bar.red.and.pred q, 1, 128, p;\n selp.u32 %0, 1, 0, q;\n}\n"
      : "=r"(r) : "r"((uint32_t)ok) : "memory");
  return r != 0;
}

// Bytes of one packed tile the loader copies (codes of K and V, metadata).
template <int D, int BITS, int FMT>
__host__ __device__ constexpr int raw_bytes() {
  return 2 * kTok * (D * BITS / 8) + (FMT == KVQ_FMT_SYMMETRIC ? 2 : 4) * 4 * D;
}

// Loader: the packed rows of tile t0 .. t0 + 63 of every plane the tile
// reads, one bulk copy per plane.  Planes hold whole 64-row tiles (their
// row counts are padded to multiples of 64), so a tile reaching past the
// stored tokens copies rows that are never used.
template <int D, int BITS, int FMT>
__device__ __forceinline__ void load_raw(const Geom& g, int b, int h, int t0, unsigned char* raw,
                                         uint64_t* bar) {
  using S = M256Layout<D, BITS>;
  constexpr uint32_t CB = kTok * S::CROW;
  mbar_expect_tx(bar, raw_bytes<D, BITS, FMT>());
  // a tile is one 64-token page of a paged cache: tok_ptr finds its rows
  bulk_copy(raw + S::RKC, tok_ptr<uint8_t>(g, KVQ_PLANE_K_CODES, b, h, t0), CB, bar);
  bulk_copy(raw + S::RVC, tok_ptr<uint8_t>(g, KVQ_PLANE_V_CODES, b, h, t0), CB, bar);
  // KIVI: two key blocks of D channels
  const __half* ks = FMT == KVQ_FMT_KIVI ? blk_ptr<__half>(g, KVQ_PLANE_K_SCALE, b, h, t0 / 32)
                                         : tok_ptr<__half>(g, KVQ_PLANE_K_SCALE, b, h, t0);
  bulk_copy(raw + S::RKS, ks, 4 * D, bar);
  if (FMT != KVQ_FMT_SYMMETRIC) {
    const __half* kz = FMT == KVQ_FMT_KIVI
                           ? blk_ptr<__half>(g, KVQ_PLANE_K_ZERO, b, h, t0 / 32)
                           : tok_ptr<__half>(g, KVQ_PLANE_K_ZERO, b, h, t0);
    bulk_copy(raw + S::RKZ, kz, 4 * D, bar);
  }
  bulk_copy(raw + S::RVS, tok_ptr<__half>(g, KVQ_PLANE_V_SCALE, b, h, t0), 4 * D, bar);
  if (FMT != KVQ_FMT_SYMMETRIC)
    bulk_copy(raw + S::RVZ, tok_ptr<__half>(g, KVQ_PLANE_V_ZERO, b, h, t0), 4 * D, bar);
}

// K: 8 channels reconstructed in fp32 and split into a bf16 high part (the
// value truncated) and the bf16 of the remainder.
__device__ __forceinline__ void split_store(const uint64_t (&k2)[4], unsigned char* hi_dst,
                                            unsigned char* lo_dst) {
  uint32_t h[4], l[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    float a, c;
    f2unpack(k2[i], a, c);
    const uint32_t ab = __float_as_uint(a) & 0xFFFF0000u, cb = __float_as_uint(c) & 0xFFFF0000u;
    h[i] = __byte_perm(ab, cb, 0x7632);
    float ra, rc;
    f2unpack(fadd2(k2[i], f2pack(-__uint_as_float(ab), -__uint_as_float(cb))), ra, rc);
    l[i] = pack_bf16(ra, rc);
  }
  *reinterpret_cast<uint4*>(hi_dst) = make_uint4(h[0], h[1], h[2], h[3]);
  *reinterpret_cast<uint4*>(lo_dst) = make_uint4(l[0], l[1], l[2], l[3]);
}

// Code e of a word of BITS-bit codes as an exact float plus 2^23.
template <int BITS>
__device__ __forceinline__ float code_biased(uint32_t w, int e) {
  constexpr uint32_t mask = (1u << BITS) - 1;
  return __uint_as_float(0x4B000000u | ((w >> (e * BITS)) & mask));
}

// Producers: reconstruct the K and V operand tiles of KV tile t0 from the
// packed tile in `raw` (tokens below tq), the KIVI residual ring (tq <= t <
// T) or zeros (t >= T).
//   K: thread (tk = tid % 64, hf = tid / 64): token tk, channels of half hf.
//   V: thread (tb = tid % 8, vq = tid / 8): tokens 8 tb .. 8 tb + 7 and
//      channels CV vq .. CV vq + CV - 1 (CV = D / 16), in half2 arithmetic,
//      stored as D rows of the transposed tile (one 16-byte chunk per row).
template <int D, int BITS, int FMT>
__device__ __forceinline__ void build_tile(const Geom& g, int b, int h, int t0, int T, int tq,
                                           int tid, const unsigned char* raw, unsigned char* kv) {
  using S = M256Layout<D, BITS>;
  constexpr bool KIVI = FMT == KVQ_FMT_KIVI;
  constexpr bool SYM = FMT == KVQ_FMT_SYMMETRIC;
  constexpr int CV = D / 16;
  constexpr int NCH = D / 16;                     // K chunks of 8 channels per thread
  constexpr int NKW = D / 2 * BITS / 32;          // K code words per thread
  const int tk = tid & 63, hf = tid >> 6;
  const int t = t0 + tk;
  // ---- K tile ----
  if (t < tq) {
    uint32_t kw[NKW];
    const unsigned char* cp = raw + S::RKC + tk * S::CROW + hf * (S::CROW / 2);
    if constexpr (NKW >= 4) {
#pragma unroll
      for (int i = 0; i < NKW / 4; ++i) {
        const uint4 u = *reinterpret_cast<const uint4*>(cp + 16 * i);
        kw[4 * i] = u.x; kw[4 * i + 1] = u.y; kw[4 * i + 2] = u.z; kw[4 * i + 3] = u.w;
      }
    } else {
      const uint2 u = *reinterpret_cast<const uint2*>(cp);
      kw[0] = u.x; kw[1] = u.y;
    }
    uint32_t ks = 0, kz = 0;                      // affine/symmetric: the half's group metadata
    if constexpr (!KIVI) {
      const unsigned char* sp = raw + S::RKS + tk * (D / 16) + hf * (D / 32);
      if constexpr (D == 128) {
        ks = *reinterpret_cast<const uint32_t*>(sp);
        if (!SYM) kz = *reinterpret_cast<const uint32_t*>(sp + (S::RKZ - S::RKS));
      } else {
        ks = *reinterpret_cast<const unsigned short*>(sp);
        if (!SYM) kz = *reinterpret_cast<const unsigned short*>(sp + (S::RKZ - S::RKS));
      }
    }
    const uint64_t bias2 = f2pack(-8388608.f, -8388608.f);
#pragma unroll
    for (int c = 0; c < NCH; ++c) {
      const int cc = hf * NCH + c;                // chunk along D
      constexpr int CB = 8 * BITS;                // code bits per chunk
      const uint32_t w = kw[(c * CB) / 32] >> ((c * CB) % 32);
      uint64_t k2[4];
      if constexpr (KIVI) {
        const unsigned char* st = raw + S::RKS + (tk >> 5) * (2 * D) + cc * 16;
        const uint4 su = *reinterpret_cast<const uint4*>(st);
        const uint4 zu = *reinterpret_cast<const uint4*>(st + (S::RKZ - S::RKS));
        const __half2* s2 = reinterpret_cast<const __half2*>(&su);
        const __half2* z2 = reinterpret_cast<const __half2*>(&zu);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const float2 sf = __half22float2(s2[i]), zf = __half22float2(z2[i]);
          const uint64_t c2 = fadd2(f2pack(code_biased<BITS>(w, 2 * i), code_biased<BITS>(w, 2 * i + 1)), bias2);
          k2[i] = ffma2(c2, f2pack(sf.x, sf.y), f2pack(zf.x, zf.y));
        }
      } else {
        const int gi = (c * 8) / 32;              // group within the half
        const __half2 s2 = *reinterpret_cast<const __half2*>(&ks);
        const __half2 z2 = *reinterpret_cast<const __half2*>(&kz);
        const float s = gi ? __high2float(s2) : __low2float(s2);
        const float m = SYM ? -(float)(1 << (BITS - 1)) * s : (gi ? __high2float(z2) : __low2float(z2));
        const uint64_t ss = f2pack(s, s), mm = f2pack(m, m);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const uint64_t c2 = fadd2(f2pack(code_biased<BITS>(w, 2 * i), code_biased<BITS>(w, 2 * i + 1)), bias2);
          k2[i] = ffma2(c2, ss, mm);
        }
      }
      unsigned char* base = kv + (cc >> 3) * (kTok * 128);
      split_store(k2, base + S::KH + sw128(tk, cc & 7), base + S::KL + sw128(tk, cc & 7));
    }
  } else {
    // KIVI residual window (full precision) or beyond the cache (zeros)
#pragma unroll
    for (int c = 0; c < NCH; ++c) {
      const int cc = hf * NCH + c;
      uint4 u = make_uint4(0, 0, 0, 0);
      if (KIVI && t < T)
        u = *reinterpret_cast<const uint4*>(
            plane_ptr<__nv_bfloat16>(g, KVQ_PLANE_K_FULL, b, h, t % g.ring, 8 * cc));
      unsigned char* base = kv + (cc >> 3) * (kTok * 128);
      *reinterpret_cast<uint4*>(base + S::KH + sw128(tk, cc & 7)) = u;
      *reinterpret_cast<uint4*>(base + S::KL + sw128(tk, cc & 7)) = make_uint4(0, 0, 0, 0);
    }
  }
  // ---- V^T tile: rows d = CV vq + e, 16-byte chunk tb (tokens 8 tb ..) ----
  const int tb = tid & 7, vq = tid >> 3;
  const int grp_v = vq * CV / 32;
  uint32_t out[CV][4];
  const __half2 bias = __float2half2_rn(1024.f);
#pragma unroll
  for (int p = 0; p < 4; ++p) {                   // token pair (2p, 2p + 1)
    uint32_t w2[2], s2u, z2u;
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      const int tv = 8 * tb + 2 * p + u;          // token within the tile
      const unsigned char* cp = raw + S::RVC + tv * S::CROW + vq * (CV * BITS / 8);
      if constexpr (CV * BITS == 32) w2[u] = *reinterpret_cast<const uint32_t*>(cp);
      else if constexpr (CV * BITS == 16) w2[u] = *reinterpret_cast<const unsigned short*>(cp);
      else w2[u] = *cp;
    }
    {
      const int tv = 8 * tb + 2 * p;
      const unsigned short* sp = reinterpret_cast<const unsigned short*>(raw + S::RVS) + tv * (D / 32) + grp_v;
      s2u = (uint32_t)sp[0] | ((uint32_t)sp[D / 32] << 16);
      if constexpr (SYM) {
        const __half2 z = __hmul2(*reinterpret_cast<const __half2*>(&s2u),
                                  __float2half2_rn(-(float)(1 << (BITS - 1))));
        z2u = *reinterpret_cast<const uint32_t*>(&z);
      } else {
        const unsigned short* zp = reinterpret_cast<const unsigned short*>(raw + S::RVZ) + tv * (D / 32) + grp_v;
        z2u = (uint32_t)zp[0] | ((uint32_t)zp[D / 32] << 16);
      }
    }
    uint32_t pw[2];
    if constexpr (CV * BITS == 32) {
      pw[0] = __byte_perm(w2[0], w2[1], 0x5410);  // low halves of both tokens
      pw[1] = __byte_perm(w2[0], w2[1], 0x7632);
    } else {
      pw[0] = (w2[0] & 0xFFFFu) | (w2[1] << 16);
      pw[1] = 0;
    }
    const __half2 s2 = *reinterpret_cast<const __half2*>(&s2u);
    const __half2 z2 = *reinterpret_cast<const __half2*>(&z2u);
#pragma unroll
    for (int e = 0; e < CV; ++e) {
      constexpr uint32_t m2 = ((1u << BITS) - 1) * 0x00010001u;
      const uint32_t x = ((pw[(e * BITS) / 16] >> ((e * BITS) % 16)) & m2) | 0x64006400u;
      const __half2 c2 = __hsub2(*reinterpret_cast<const __half2*>(&x), bias);
      const __half2 v2 = __hfma2(s2, c2, z2);
      out[e][p] = *reinterpret_cast<const uint32_t*>(&v2);
    }
  }
  // tokens of the KIVI residual window, or beyond the cache, replace theirs
  const int tv0 = t0 + 8 * tb;
  if (tv0 + 7 >= tq) {
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int tv = tv0 + i;
      if (tv < tq) continue;
      __nv_bfloat16 vals[CV];
      if (KIVI && tv < T) {
        const __nv_bfloat16* src = plane_ptr<__nv_bfloat16>(g, KVQ_PLANE_V_FULL, b, h, tv % g.ring, vq * CV);
        if constexpr (CV == 8) {
          const uint4 u = *reinterpret_cast<const uint4*>(src);
          memcpy(vals, &u, sizeof(vals));
        } else {
          const uint2 u = *reinterpret_cast<const uint2*>(src);
          memcpy(vals, &u, sizeof(vals));
        }
      } else {
#pragma unroll
        for (int e = 0; e < CV; ++e) vals[e] = __float2bfloat16_rn(0.f);
      }
#pragma unroll
      for (int e = 0; e < CV; ++e) {
        const uint32_t hv = __half_as_ushort(__float2half_rn(__bfloat162float(vals[e])));
        out[e][i >> 1] = (i & 1) ? ((out[e][i >> 1] & 0xFFFFu) | (hv << 16))
                                 : ((out[e][i >> 1] & 0xFFFF0000u) | hv);
      }
    }
  }
#pragma unroll
  for (int e = 0; e < CV; ++e)
    *reinterpret_cast<uint4*>(kv + S::VT + sw128(CV * vq + e, tb)) =
        make_uint4(out[e][0], out[e][1], out[e][2], out[e][3]);
}

template <int D, int BITS, int FMT>
__global__ void __launch_bounds__(kThreads, 1)
attend_prefill_m256_kernel(Geom g, const __nv_bfloat16* __restrict__ q, int L, float scale,
                           __nv_bfloat16* __restrict__ out, int nq, int* err) {
  pdl_wait();
  pdl_trigger();
  using S = M256Layout<D, BITS>;
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ uint64_t raw_full[kRaw], raw_free[kRaw], kv_full[kKvBufs], kv_free[kKvBufs],
      s_full[2][2], p_full[2][2], s_free[2][2], done_bar;
  __shared__ uint32_t tmem_base;
  __shared__ int abort_flag;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nqt = gridDim.x;
  const int qtile = nqt - 1 - blockIdx.x;              // longest first
  const int hkv = blockIdx.y, b = blockIdx.z;
  const int grp = g.Hq / g.H;
  const int T = seq_tokens(g, b);
  const int tq = FMT == KVQ_FMT_KIVI ? kivi_tq(T, g.R, g.G) : T;
  // a ragged cache's sequence b attends the rows of its last append
  const int Lb = g.layout == KVQ_LAYOUT_UNIFORM ? L : g.seq_new[b];
  const int q0 = qtile * nq;
  if (q0 >= Lb) return;                                // no query of this sequence here
  const int nql = min(nq, Lb - q0);
  const int pos_first = T - Lb + q0;
  const int t_end = pos_first + nql;                   // keys [0, t_end)
  const int ntiles = (t_end + kTok - 1) / kTok;
  volatile int* abort = &abort_flag;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kRaw; ++i) {
      mbar_init(&raw_full[i], 1);
      mbar_init(&raw_free[i], 128);
    }
    for (int i = 0; i < kKvBufs; ++i) {
      mbar_init(&kv_full[i], 128);
      mbar_init(&kv_free[i], 1);
    }
    for (int x = 0; x < 2; ++x)
      for (int i = 0; i < 2; ++i) {
        mbar_init(&s_full[x][i], 1);
        mbar_init(&p_full[x][i], 128);
        mbar_init(&s_free[x][i], 1);
      }
    mbar_init(&done_bar, 1);
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 12) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 512;"
                 ::"r"(smem_u32(&tmem_base)));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  // queries -> the swizzled Q tiles (softmax threads, one row each)
  const int row = threadIdx.x;                          // 0..255 for the softmax roles
  int pos = -1;
  if (warp < 8) {
    const int hl = row / nq, qi = row % nq;
    const bool valid = hl < grp && qi < nql;
    if (valid) pos = pos_first + qi;
    const __nv_bfloat16* src = q + (((int64_t)b * g.Hq + hkv * grp + hl) * L + q0 + qi) * D;
    unsigned char* qt = smem + S::Q_OFF + (row >> 7) * S::QT;
    const int r = row & 127;
#pragma unroll
    for (int c = 0; c < D / 8; ++c) {
      uint4 v = make_uint4(0, 0, 0, 0);
      if (valid) v = *reinterpret_cast<const uint4*>(src + 8 * c);
      *reinterpret_cast<uint4*>(qt + (c >> 3) * (kM * 128) + sw128(r, c & 7)) = v;
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base;

  if (warp == 13) {
    // ---------------- loader: packed tiles into the raw ring ----------------
    if (lane == 0) {
      int issued = 0;
      for (int j = 0; j < ntiles; ++j) {
        const int st = j % kRaw;
        if (j >= kRaw && !mbar_wait_or_abort(&raw_free[st], ((j - kRaw) / kRaw) & 1, abort)) break;
        load_raw<D, BITS, FMT>(g, b, hkv, j * kTok, smem + S::RAW_OFF + st * S::RAW_B,
                               &raw_full[st]);
        issued = j + 1;
      }
      // no copy may still be landing in shared memory when the CTA exits
      // (after a timeout the producers stop consuming): wait, bounded, for
      // the last tile issued on each stage
      for (int t = issued > kRaw ? issued - kRaw : 0; t < issued; ++t)
        if (!mbar_wait(&raw_full[t % kRaw], (t / kRaw) & 1)) *abort = 1;
    }
  } else if (warp >= 8 && warp < 12) {
    // ---------------- producers: reconstruct K and V tiles ----------------
    const int tid = threadIdx.x - 256;
    for (int j = 0; j < ntiles; ++j) {
      const int st = j % kRaw, kb = j % kKvBufs;
      bool ok = mbar_wait_or_abort(&raw_full[st], (j / kRaw) & 1, abort);
      ok = ok && (j < kKvBufs ||
                  mbar_wait_or_abort(&kv_free[kb], ((j - kKvBufs) / kKvBufs) & 1, abort));
      if (!producers_all(ok)) break;
      unsigned char* kv = smem + S::KV_OFF + kb * S::KV_B;
      build_tile<D, BITS, FMT>(g, b, hkv, j * kTok, T, tq, tid, smem + S::RAW_OFF + st * S::RAW_B, kv);
      mbar_arrive(&raw_free[st]);
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      mbar_arrive(&kv_full[kb]);
    }
  } else if (warp == 12) {
    // ---------------- MMA issuer ----------------
    // Issues, as soon as each is ready: Q K^T of the next tile for both
    // query tiles (its K/V tile built, the S buffer's previous P V done),
    // and P V of each query tile's next tile (its P written).  S runs one
    // tile ahead of the softmax threads; the tensor pipe executes in issue
    // order.  The whole warp runs the loop (its values stay warp-uniform)
    // and one elected lane issues the MMAs and their commits.  Descriptors
    // are formed once: a K step of 16 elements advances the start address by
    // 32 bytes (2 in the descriptor's 16-byte units).
    constexpr uint32_t id_qk = idesc_bf16(kM, kTok);
    constexpr uint32_t id_pv = idesc_f16(kM, D);
    const uint64_t qdesc0 = sw128_desc(smem + S::Q_OFF);
    const uint64_t kvdesc0 = sw128_desc(smem + S::KV_OFF);   // K/V buffer b: + b KV_B / 16
    const bool leader = elect_one();
    int nqk = 0, npv[2] = {0, 0};
    long idle = 0;
    uint64_t idle_since = 0;
    while (npv[0] < ntiles || npv[1] < ntiles) {
      bool progressed = false;
      if (nqk < ntiles && nqk <= min(npv[0], npv[1]) + 1) {
        const int kb = nqk % kKvBufs, bf = nqk & 1;
        const uint32_t fpar = (nqk >= 2) ? ((nqk - 2) >> 1) & 1 : 0;
        bool ready = false;
        if (lane == 0)
          ready = mbar_test(&kv_full[kb], (nqk / kKvBufs) & 1) &&
                  (nqk < 2 || (mbar_test(&s_free[0][bf], fpar) && mbar_test(&s_free[1][bf], fpar)));
        if (__shfl_sync(0xffffffffu, ready, 0)) {
          tc_fence_after();
          if (leader) {
#pragma unroll
            for (int x = 0; x < 2; ++x) {
              const uint32_t ts = tmem + x * 128 + bf * kTok;
#pragma unroll
              for (int kk = 0; kk < D / 16; ++kk) {
                // Q atom: 128 rows x 128 B (1024 units); K atom: 64 rows x 128 B (512 units)
                const uint64_t qd = qdesc0 + (uint64_t)(x * (S::QT >> 4) + (kk >> 2) * 1024 + (kk & 3) * 2);
                const uint64_t kd = kvdesc0 + (uint64_t)(kb * (S::KV_B >> 4) + (kk >> 2) * 512 + (kk & 3) * 2);
                umma_a_fill(ts, qd, kd + (S::KH >> 4), id_qk, kk > 0);   // Q read once
                umma_a_lastuse(ts, qd, kd + (S::KL >> 4), id_qk, 1);     // for K hi and lo
              }
              umma_commit(&s_full[x][bf]);
            }
          }
          __syncwarp();
          ++nqk;
          progressed = true;
        }
      }
#pragma unroll
      for (int x = 0; x < 2; ++x) {
        const int j = npv[x];
        if (j >= nqk) continue;
        const int bf = j & 1;
        bool ready = false;
        if (lane == 0) ready = mbar_test(&p_full[x][bf], (j >> 1) & 1);
        if (!__shfl_sync(0xffffffffu, ready, 0)) continue;
        tc_fence_after();
        const int kb = j % kKvBufs;
        if (leader) {
          const uint32_t tp = tmem + x * 128 + bf * kTok;   // P (fp16 pairs) over S's columns
          const uint32_t to = tmem + 256 + x * D;
#pragma unroll
          for (int kk = 0; kk < kTok / 16; ++kk)
            umma_ts(to, tp + kk * 8, kvdesc0 + (uint64_t)(kb * (S::KV_B >> 4) + (S::VT >> 4) + kk * 2),
                    id_pv, (j > 0 || kk > 0) ? 1u : 0u);
          umma_commit(&s_free[x][bf]);           // S/P buffer free, and O holds tile j
          if (npv[x ^ 1] > j) umma_commit(&kv_free[kb]);   // both query tiles done with it
        }
        __syncwarp();
        ++npv[x];
        progressed = true;
      }
      if (progressed) {
        idle = 0;
      } else {
        if (idle == 0) idle_since = global_ns();
        __nanosleep(20);
        const bool stop = (++idle & 63) == 0 && (*abort || global_ns() - idle_since > kWaitNs);
        if (__shfl_sync(0xffffffffu, stop, 0)) break;   // the whole warp leaves together
      }
    }
    if (lane == 0 && (npv[0] < ntiles || npv[1] < ntiles)) *abort = 1;
    if (leader) umma_commit(&done_bar);        // every MMA issued above has completed
    if (lane == 0 && !mbar_wait(&done_bar, 0)) *abort = 1;
    __syncwarp();
  } else if (warp < 8) {
    // ---------------- softmax: one row per thread ----------------
    const int x = warp >> 2;                   // query tile
    const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
    const uint32_t s_col = tmem + lane_base + x * 128;
    const uint32_t o_col = tmem + lane_base + 256 + x * D;
    const float c2 = scale * 1.4426950408889634f;   // scores in log2 units
    const uint64_t c22 = f2pack(c2, c2);
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    for (int j = 0; j < ntiles; ++j) {
      const int bf = j & 1, t0 = j * kTok;
      if (!warp_wait(&s_full[x][bf], (j >> 1) & 1, abort)) {
        ok = false;
        break;
      }
      tc_fence_after();
      uint32_t sr[kTok];
#pragma unroll
      for (int c = 0; c < kTok; c += 16) tmem_ld16_nowait(s_col + bf * kTok + c, sr + c);
      tmem_wait_ld();
      const bool full = t0 + kTok - 1 <= pos;  // no key of the tile is masked
      if (!full) {
#pragma unroll
        for (int i = 0; i < kTok; ++i)
          if (t0 + i > pos) sr[i] = __float_as_uint(-INFINITY);
      }
      // row maximum: four independent chains of three-input maxima over
      // 16 scores each
      float mx4[4];
#pragma unroll
      for (int a = 0; a < 4; ++a) {
        const uint32_t* v = sr + 16 * a;
        float mv = fmax3(__uint_as_float(v[0]), __uint_as_float(v[1]), __uint_as_float(v[2]));
#pragma unroll
        for (int k = 3; k < 15; k += 2)
          mv = fmax3(mv, __uint_as_float(v[k]), __uint_as_float(v[k + 1]));
        mx4[a] = fmaxf(mv, __uint_as_float(v[15]));
      }
      const float mx = fmaxf(fmaxf(mx4[0], mx4[1]), fmaxf(mx4[2], mx4[3]));
      const float m_new = fmaxf(m, mx * c2);   // (c2 > 0: the maximum commutes)
      if (j == 0) {
        m = m_new;
      } else if (__any_sync(0xffffffffu, m_new > m + kRescale)) {
        // O is rewritten: the P V of tile j - 1 must have completed
        if (!warp_wait(&s_free[x][(j - 1) & 1], ((j - 1) >> 1) & 1, abort)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const float alpha = m_new > m ? ex2_approx(m - m_new) : 1.f;
        if (m_new > m) {
          l *= alpha;
          m = m_new;
        }
#pragma unroll 1
        for (int c = 0; c < D; c += 16) {
          uint32_t o[16];
          tmem_ld16_nowait(o_col + c, o);
          tmem_wait_ld();
#pragma unroll
          for (int i = 0; i < 16; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * alpha);
          tmem_st16(o_col + c, o);
        }
      }
      // P = 2^(s c2 - m) as fp16 pairs over the first 32 columns of this S
      // buffer (masked keys hold -inf: 2^-inf = 0; a row without any visible
      // key so far has m = -inf and keeps P = 0)
      const bool live = m != -INFINITY;
      const uint64_t negm = f2pack(-m, -m);
      uint64_t sum2 = f2pack(0.f, 0.f);
      uint32_t pk[kTok / 2];
#pragma unroll
      for (int i = 0; i < kTok; i += 2) {
        float a0, a1;
        f2unpack(ffma2(f2pack(__uint_as_float(sr[i]), __uint_as_float(sr[i + 1])), c22, negm), a0, a1);
        float p0 = ex2_approx(a0), p1 = ex2_approx(a1);
        if (!live) p0 = p1 = 0.f;
        sum2 = fadd2(sum2, f2pack(p0, p1));
        pk[i / 2] = pack_h2(p0, p1);
      }
      tmem_st16(s_col + bf * kTok, pk);
      tmem_st16(s_col + bf * kTok + 16, pk + 16);
      float s0, s1;
      f2unpack(sum2, s0, s1);
      l += s0 + s1;
      tmem_wait_st();
      tc_fence_before();
      mbar_arrive(&p_full[x][bf]);
    }
    // ---------------- epilogue ----------------
    if (ok && ntiles > 0 &&
        !warp_wait(&s_free[x][(ntiles - 1) & 1], ((ntiles - 1) >> 1) & 1, abort))
      ok = false;
    if (__all_sync(0xffffffffu, ok && !*abort)) {
      tc_fence_after();
      const float inv = l > 0.f ? 1.f / l : 0.f;
      const int hl = row / nq, qi = row % nq;
      __nv_bfloat16* dst = out + (((int64_t)b * g.Hq + hkv * grp + hl) * L + q0 + qi) * D;
#pragma unroll 1
      for (int c = 0; c < D; c += 16) {
        uint32_t o[16];
        tmem_ld16_nowait(o_col + c, o);
        tmem_wait_ld();
        if (pos >= 0) {
          uint32_t w[8];
#pragma unroll
          for (int i = 0; i < 8; ++i)
            w[i] = pack_bf16(__uint_as_float(o[2 * i]) * inv, __uint_as_float(o[2 * i + 1]) * inv);
          *reinterpret_cast<uint4*>(dst + c) = make_uint4(w[0], w[1], w[2], w[3]);
          *reinterpret_cast<uint4*>(dst + c + 8) = make_uint4(w[4], w[5], w[6], w[7]);
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0 && *abort) atomicOr(err, 8);
  if (warp == 12) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 512;" ::"r"(tmem));
  }
}

template <int D, int BITS, int FMT>
cudaError_t launch_m256(const Geom& g, const void* q, int L, float scale, void* out, int* err,
                        cudaStream_t s) {
  auto kern = attend_prefill_m256_kernel<D, BITS, FMT>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       M256Layout<D, BITS>::ALLOC);
  if (e != cudaSuccess) return e;
  const int nq = kRowsCta / (g.Hq / g.H);
  dim3 grid((L + nq - 1) / nq, g.H, g.B);
  launch_pdl(kern, dim3(grid), dim3(kThreads), (size_t)M256Layout<D, BITS>::ALLOC, s, g,
             reinterpret_cast<const __nv_bfloat16*>(q), L, scale,
             reinterpret_cast<__nv_bfloat16*>(out), nq, err);
  return cudaGetLastError();
}

template <int D>
cudaError_t launch_m256_d(const Geom& g, const void* q, int L, float scale, void* out, int* err,
                          cudaStream_t s) {
  if (g.fmt == KVQ_FMT_KIVI)
    return g.kb == 4 ? launch_m256<D, 4, KVQ_FMT_KIVI>(g, q, L, scale, out, err, s)
                     : launch_m256<D, 2, KVQ_FMT_KIVI>(g, q, L, scale, out, err, s);
  if (g.fmt == KVQ_FMT_SYMMETRIC)
    return g.kb == 4 ? launch_m256<D, 4, KVQ_FMT_SYMMETRIC>(g, q, L, scale, out, err, s)
                     : launch_m256<D, 2, KVQ_FMT_SYMMETRIC>(g, q, L, scale, out, err, s);
  return g.kb == 4 ? launch_m256<D, 4, KVQ_FMT_AFFINE>(g, q, L, scale, out, err, s)
                   : launch_m256<D, 2, KVQ_FMT_AFFINE>(g, q, L, scale, out, err, s);
}

}  // namespace

// bf16 affine/symmetric/KIVI caches with equal 2- or 4-bit key and value
// codes, G = 32 (KIVI: 32-token key blocks), head_dim 64 or 128, GQA group <= 256.
bool prefill_m256_supported(const Geom& g) {
  const bool fmt_ok = g.fmt == KVQ_FMT_AFFINE || g.fmt == KVQ_FMT_SYMMETRIC || g.fmt == KVQ_FMT_KIVI;
  return fmt_ok && g.act == KVQ_BF16 && (g.D == 64 || g.D == 128) && g.G == 32 && g.kb == g.vb &&
         (g.kb == 2 || g.kb == 4) && g.Hq / g.H <= kRowsCta;
}

cudaError_t launch_prefill_m256(const Geom& g, const void* q, int L, float scale, void* out,
                                int* err, cudaStream_t s) {
  if (g.D == 64) return launch_m256_d<64>(g, q, L, scale, out, err, s);
  return launch_m256_d<128>(g, q, L, scale, out, err, s);
}

}  // namespace kvq
