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
//   issuer (warp 12, one thread): S_X = Q_X K_hi^T + Q_X K_lo^T for X = A, B
//     into double-buffered TMEM tiles (128 x 64 fp32), then, one KV tile
//     behind, O_X += P_X V into a TMEM accumulator (128 x D fp32) per query
//     tile; completions are signalled by tcgen05.commit on mbarriers;
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
constexpr int kThreads = 13 * 32;    // 8 softmax warps, 4 producer warps, 1 issuer warp
constexpr float kRescale = 8.f;      // log2 growth of a row maximum that forces a rescale

// Shared memory (bytes from a 1024-aligned base).
template <int D>
struct M256Layout {
  static constexpr int QT = kM * D * 2;             // one query tile: D/64 atoms of 16 KB
  static constexpr int Q_OFF = 0;
  static constexpr int KV_OFF = 2 * QT;
  static constexpr int KH = 0;                      // K hi: D/64 atoms of 64 rows x 128 B
  static constexpr int KL = kTok * D * 2;           // K lo: the same
  static constexpr int VT = 2 * kTok * D * 2;       // V^T: D rows x 128 B (64 tokens)
  static constexpr int KV_B = VT + D * 128;
  static constexpr int P_OFF = KV_OFF + 2 * KV_B;   // P of tile A, then of tile B
  static constexpr int P_B = kM * kTok * 2;         // 128 rows x 128 B (fp16)
  static constexpr int SC_OFF = P_OFF + 2 * P_B;    // KIVI key block scales, 2 buffers
  static constexpr int SC_B = 2 * 2 * D * 2;        // 2 blocks x (scale, zero) x D fp16
  static constexpr int TOTAL = SC_OFF + 2 * SC_B;
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

// What one producer thread loads for one KV tile ahead of its use.
//   K: token tk of the tile, channel half hf (D/2 channels): its code words,
//      and (affine/symmetric) the token's fp16 group scales and offsets of
//      that half; (KIVI) one 16-byte piece of the tile's per-channel block
//      scales, staged in shared memory for all producers.
//   V: tokens 8 tb .. 8 tb + 7 of the tile, channels CV vq .. CV vq + CV - 1
//      (CV = D/16): each token's code word of those channels and its group
//      scale and offset, paired by token for half2 arithmetic.
template <int D, int BITS>
struct TileCodes {
  static constexpr int NKW = D / 2 * BITS / 32;      // K code words per thread
  uint32_t kw[NKW];
  uint32_t ks, kz;                                   // fp16 pairs (groups of the half)
  uint4 stage;                                       // KIVI block scales piece
  uint32_t vw[8];                                    // V code word per token
  uint32_t vs[4], vz[4];                             // half2 (token 2i, 2i + 1)
};

// Where a tile's tokens come from: codes (t < tq), the KIVI residual ring
// (tq <= t < T) or nothing (t >= T: zeros).
template <int D, int BITS, int FMT>
__device__ __forceinline__ void load_tile(const Geom& g, int b, int h, int t0, int T, int tq,
                                          int tid, TileCodes<D, BITS>& r) {
  constexpr bool KIVI = FMT == KVQ_FMT_KIVI;
  constexpr bool SYM = FMT == KVQ_FMT_SYMMETRIC;
  constexpr int CV = D / 16;
  const int tk = tid & 63, hf = tid >> 6;
  const int t = t0 + tk;
  // ---- K ----
  if (t < tq) {
    const uint8_t* row = plane_ptr<uint8_t>(g, KVQ_PLANE_K_CODES, b, h, t) + hf * (D / 2 * BITS / 8);
    if constexpr (TileCodes<D, BITS>::NKW >= 4) {
#pragma unroll
      for (int i = 0; i < TileCodes<D, BITS>::NKW / 4; ++i) {
        const uint4 u = __ldg(reinterpret_cast<const uint4*>(row) + i);
        r.kw[4 * i] = u.x; r.kw[4 * i + 1] = u.y; r.kw[4 * i + 2] = u.z; r.kw[4 * i + 3] = u.w;
      }
    } else {
      const uint2 u = __ldg(reinterpret_cast<const uint2*>(row));
      r.kw[0] = u.x; r.kw[1] = u.y;
    }
    if constexpr (!KIVI) {
      // groups of 32 channels: D/64 groups in this half
      const __half* sp = plane_ptr<__half>(g, KVQ_PLANE_K_SCALE, b, h, t, hf * (D / 64));
      if constexpr (D == 128) {
        r.ks = __ldg(reinterpret_cast<const uint32_t*>(sp));
        r.kz = SYM ? 0u : __ldg(reinterpret_cast<const uint32_t*>(
                              plane_ptr<__half>(g, KVQ_PLANE_K_ZERO, b, h, t, hf * 2)));
      } else {
        r.ks = __half_as_ushort(__ldg(sp));
        r.kz = SYM ? 0u : __half_as_ushort(__ldg(plane_ptr<__half>(g, KVQ_PLANE_K_ZERO, b, h, t, hf)));
      }
    }
  } else {
#pragma unroll
    for (int i = 0; i < TileCodes<D, BITS>::NKW; ++i) r.kw[i] = 0;
    r.ks = r.kz = 0;
  }
  if constexpr (KIVI) {
    // staged block scales: [block 0, 1][scale, zero][D] fp16 = 4 D / 8 pieces
    r.stage = make_uint4(0, 0, 0, 0);
    if (tid < 4 * D / 8) {
      const int blk = tid / (2 * D / 8), rem = tid % (2 * D / 8);
      const int sz = rem / (D / 8), ch = rem % (D / 8);
      const int tb0 = t0 + 32 * blk;
      if (tb0 < tq)
        r.stage = __ldg(reinterpret_cast<const uint4*>(
            plane_ptr<__half>(g, sz ? KVQ_PLANE_K_ZERO : KVQ_PLANE_K_SCALE, b, h, tb0 / 32, 8 * ch)));
    }
  }
  // ---- V ----
  const int tb = tid & 7, vq = tid >> 3;
  const int grp_v = vq * CV / 32;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int tv = t0 + 8 * tb + i;
    uint32_t w = 0;
    __half s = __ushort_as_half(0), z = __ushort_as_half(0);
    if (tv < tq) {
      const uint8_t* row = plane_ptr<uint8_t>(g, KVQ_PLANE_V_CODES, b, h, tv) + vq * (CV * BITS / 8);
      if constexpr (CV * BITS == 32) w = __ldg(reinterpret_cast<const uint32_t*>(row));
      else if constexpr (CV * BITS == 16) w = __ldg(reinterpret_cast<const unsigned short*>(row));
      else w = __ldg(row);
      s = __ldg(plane_ptr<__half>(g, KVQ_PLANE_V_SCALE, b, h, tv, grp_v));
      z = SYM ? __hmul(s, __float2half_rn(-(float)(1 << (BITS - 1))))
              : __ldg(plane_ptr<__half>(g, KVQ_PLANE_V_ZERO, b, h, tv, grp_v));
    }
    r.vw[i] = w;
    if (i & 1) {
      r.vs[i >> 1] |= (uint32_t)__half_as_ushort(s) << 16;
      r.vz[i >> 1] |= (uint32_t)__half_as_ushort(z) << 16;
    } else {
      r.vs[i >> 1] = __half_as_ushort(s);
      r.vz[i >> 1] = __half_as_ushort(z);
    }
  }
}

// K: 8 channels (chunk c of this thread's half) reconstructed in fp32 and
// split into bf16 high (truncation) and low (rounded remainder) parts.
__device__ __forceinline__ void split_store(float (&k)[8], unsigned char* hi_dst,
                                            unsigned char* lo_dst) {
  uint32_t h[4], l[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint32_t a = __float_as_uint(k[2 * i]), c = __float_as_uint(k[2 * i + 1]);
    h[i] = __byte_perm(a, c, 0x7632);
    const float ra = k[2 * i] - __uint_as_float(a & 0xFFFF0000u);
    const float rc = k[2 * i + 1] - __uint_as_float(c & 0xFFFF0000u);
    l[i] = pack_bf16(ra, rc);
  }
  *reinterpret_cast<uint4*>(hi_dst) = make_uint4(h[0], h[1], h[2], h[3]);
  *reinterpret_cast<uint4*>(lo_dst) = make_uint4(l[0], l[1], l[2], l[3]);
}

template <int BITS>
__device__ __forceinline__ float code_f(uint32_t w, int e) {
  constexpr uint32_t mask = (1u << BITS) - 1;
  return __uint_as_float(0x4B000000u | ((w >> (e * BITS)) & mask)) - 8388608.f;
}

template <int D, int BITS, int FMT>
__device__ __forceinline__ void build_tile(const Geom& g, int b, int h, int t0, int T, int tq,
                                           int tid, const TileCodes<D, BITS>& r,
                                           const unsigned char* stage, unsigned char* kv) {
  using S = M256Layout<D>;
  constexpr bool KIVI = FMT == KVQ_FMT_KIVI;
  constexpr bool SYM = FMT == KVQ_FMT_SYMMETRIC;
  constexpr int CV = D / 16;
  constexpr int NCH = D / 16;                     // K chunks of 8 channels per thread
  const int tk = tid & 63, hf = tid >> 6;
  const int t = t0 + tk;
  // ---- K tile ----
  if (!KIVI || t < tq) {
#pragma unroll
    for (int c = 0; c < NCH; ++c) {
      const int cc = hf * NCH + c;                // chunk along D
      constexpr int CB = 8 * BITS;                // code bits per chunk
      const uint32_t w = (r.kw[(c * CB) / 32] >> ((c * CB) % 32));
      float k[8];
      if constexpr (KIVI) {
        const unsigned char* st = stage + (tk >> 5) * (4 * D) + cc * 16;
        const uint4 su = *reinterpret_cast<const uint4*>(st);
        const uint4 zu = *reinterpret_cast<const uint4*>(st + 2 * D);
        const __half2* s2 = reinterpret_cast<const __half2*>(&su);
        const __half2* z2 = reinterpret_cast<const __half2*>(&zu);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const float2 sf = __half22float2(s2[i]), zf = __half22float2(z2[i]);
          k[2 * i] = fmaf(code_f<BITS>(w, 2 * i), sf.x, zf.x);
          k[2 * i + 1] = fmaf(code_f<BITS>(w, 2 * i + 1), sf.y, zf.y);
        }
      } else {
        const int gi = (c * 8) / 32;              // group within the half
        const __half2 s2 = *reinterpret_cast<const __half2*>(&r.ks);
        const __half2 z2 = *reinterpret_cast<const __half2*>(&r.kz);
        const float s = gi ? __high2float(s2) : __low2float(s2);
        const float m = SYM ? -(float)(1 << (BITS - 1)) * s : (gi ? __high2float(z2) : __low2float(z2));
#pragma unroll
        for (int e = 0; e < 8; ++e) k[e] = fmaf(code_f<BITS>(w, e), s, m);
      }
      unsigned char* base = kv + (cc >> 3) * (kTok * 128);
      split_store(k, base + S::KH + sw128(tk, cc & 7), base + S::KL + sw128(tk, cc & 7));
    }
  } else {
    // KIVI residual window (full precision) or beyond the cache (zeros)
#pragma unroll
    for (int c = 0; c < NCH; ++c) {
      const int cc = hf * NCH + c;
      uint4 u = make_uint4(0, 0, 0, 0);
      if (t < T)
        u = *reinterpret_cast<const uint4*>(
            plane_ptr<__nv_bfloat16>(g, KVQ_PLANE_K_FULL, b, h, t % g.ring, 8 * cc));
      unsigned char* base = kv + (cc >> 3) * (kTok * 128);
      *reinterpret_cast<uint4*>(base + S::KH + sw128(tk, cc & 7)) = u;
      *reinterpret_cast<uint4*>(base + S::KL + sw128(tk, cc & 7)) = make_uint4(0, 0, 0, 0);
    }
  }
  // ---- V^T tile: rows d = CV vq + e, 16-byte chunk tb (tokens 8 tb ..) ----
  const int tb = tid & 7, vq = tid >> 3;
  uint32_t out[CV][4];
  const __half2 bias = __float2half2_rn(1024.f);
#pragma unroll
  for (int p = 0; p < 4; ++p) {                   // token pair (2p, 2p + 1)
    const uint32_t w0 = r.vw[2 * p], w1 = r.vw[2 * p + 1];
    uint32_t pw[2];
    if constexpr (CV * BITS == 32) {
      pw[0] = __byte_perm(w0, w1, 0x5410);        // low halves: channels 0 .. 16/BITS - 1
      pw[1] = __byte_perm(w0, w1, 0x7632);
    } else {
      pw[0] = (w0 & 0xFFFFu) | (w1 << 16);
      pw[1] = 0;
    }
    const __half2 s2 = *reinterpret_cast<const __half2*>(&r.vs[p]);
    const __half2 z2 = *reinterpret_cast<const __half2*>(&r.vz[p]);
#pragma unroll
    for (int e = 0; e < CV; ++e) {
      constexpr uint32_t m2 = ((1u << BITS) - 1) * 0x00010001u;
      const uint32_t x = ((pw[(e * BITS) / 16] >> ((e * BITS) % 16)) & m2) | 0x64006400u;
      const __half2 c2 = __hsub2(*reinterpret_cast<const __half2*>(&x), bias);
      const __half2 v2 = __hfma2(s2, c2, z2);
      out[e][p] = *reinterpret_cast<const uint32_t*>(&v2);
    }
  }
  if constexpr (KIVI) {
    // tokens of the residual window (or beyond the cache) replace their pair halves
    const int tv0 = t0 + 8 * tb;
    if (tv0 + 7 >= tq) {
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int tv = tv0 + i;
        if (tv < tq) continue;
        uint4 raw[CV / 8 > 0 ? CV / 8 : 1];
        __nv_bfloat16 vals[CV];
        if (tv < T) {
          const __nv_bfloat16* src = plane_ptr<__nv_bfloat16>(g, KVQ_PLANE_V_FULL, b, h, tv % g.ring, vq * CV);
          if constexpr (CV == 8) {
            raw[0] = *reinterpret_cast<const uint4*>(src);
            memcpy(vals, raw, sizeof(vals));
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
  using S = M256Layout<D>;
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ uint64_t kv_full[2], kv_free[2], s_full[2][2], s_free[2][2], p_full[2], pv_done[2],
      done_bar;
  __shared__ uint32_t tmem_base;
  __shared__ int abort_flag;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nqt = gridDim.x;
  const int qtile = nqt - 1 - blockIdx.x;              // longest first
  const int hkv = blockIdx.y, b = blockIdx.z;
  const int grp = g.Hq / g.H;
  const int T = cache_tokens(g);
  const int tq = FMT == KVQ_FMT_KIVI ? kivi_tq(T, g.R, g.G) : T;
  const int q0 = qtile * nq;
  const int nql = min(nq, L - q0);
  const int pos_first = T - L + q0;
  const int t_end = pos_first + nql;                   // keys [0, t_end)
  const int ntiles = (t_end + kTok - 1) / kTok;
  volatile int* abort = &abort_flag;

  if (threadIdx.x == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(&kv_full[i], 128);
      mbar_init(&kv_free[i], 1);
      mbar_init(&p_full[i], 128);
      mbar_init(&pv_done[i], 1);
      for (int x = 0; x < 2; ++x) {
        mbar_init(&s_full[x][i], 1);
        mbar_init(&s_free[x][i], 128);
      }
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

  if (warp >= 8 && warp < 12) {
    // ---------------- producers: reconstruct K and V tiles ----------------
    const int tid = threadIdx.x - 256;
    TileCodes<D, BITS> cur, nxt;
    load_tile<D, BITS, FMT>(g, b, hkv, 0, T, tq, tid, cur);
    for (int j = 0; j < ntiles; ++j) {
      const int bf = j & 1;
      unsigned char* stage = smem + S::SC_OFF + bf * S::SC_B;
      if (FMT == KVQ_FMT_KIVI && tid < 4 * D / 8)
        *reinterpret_cast<uint4*>(stage + 16 * tid) = cur.stage;
      const bool ok = j < 2 || mbar_wait_or_abort(&kv_free[bf], ((j - 2) >> 1) & 1, abort);
      if (!producers_all(ok)) break;                  // also publishes the staged scales
      if (j + 1 < ntiles) load_tile<D, BITS, FMT>(g, b, hkv, (j + 1) * kTok, T, tq, tid, nxt);
      unsigned char* kv = smem + S::KV_OFF + bf * S::KV_B;
      build_tile<D, BITS, FMT>(g, b, hkv, j * kTok, T, tq, tid, cur, stage, kv);
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      mbar_arrive(&kv_full[bf]);
      cur = nxt;
    }
  } else if (warp == 12 && lane == 0) {
    // ---------------- MMA issuer ----------------
    constexpr uint32_t id_qk = idesc_bf16(kM, kTok);
    constexpr uint32_t id_pv = idesc_f16(kM, D);
    bool ok = true;
    for (int j = 0; j <= ntiles && ok; ++j) {
      if (j < ntiles) {
        const int bf = j & 1;
        if (!mbar_wait_or_abort(&kv_full[bf], (j >> 1) & 1, abort)) break;
        const unsigned char* kv = smem + S::KV_OFF + bf * S::KV_B;
        for (int x = 0; x < 2 && ok; ++x) {
          if (j >= 2 && !mbar_wait_or_abort(&s_free[x][bf], ((j - 2) >> 1) & 1, abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t ts = tmem + x * 128 + bf * kTok;
          const unsigned char* qt = smem + S::Q_OFF + x * S::QT;
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const int a = kk >> 2, k4 = (kk & 3) * 32;
            const uint64_t qd = sw128_desc(qt + a * (kM * 128) + k4);
            umma(ts, qd, sw128_desc(kv + S::KH + a * (kTok * 128) + k4), id_qk, kk > 0);
            umma(ts, qd, sw128_desc(kv + S::KL + a * (kTok * 128) + k4), id_qk, 1);
          }
          umma_commit(&s_full[x][bf]);
        }
      }
      if (j >= 1 && ok) {
        const int jj = j - 1, bf = jj & 1;
        const unsigned char* kv = smem + S::KV_OFF + bf * S::KV_B;
        for (int x = 0; x < 2; ++x) {
          if (!mbar_wait_or_abort(&p_full[x], jj & 1, abort)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const unsigned char* p = smem + S::P_OFF + x * S::P_B;
          const uint32_t to = tmem + 256 + x * D;
#pragma unroll
          for (int kk = 0; kk < kTok / 16; ++kk)
            umma(to, sw128_desc(p + kk * 32), sw128_desc(kv + S::VT + kk * 32), id_pv,
                 (jj > 0 || kk > 0) ? 1u : 0u);
          umma_commit(&pv_done[x]);
        }
        if (ok) umma_commit(&kv_free[bf]);
      }
    }
    umma_commit(&done_bar);                    // every MMA issued above has completed
    if (!mbar_wait(&done_bar, 0)) *abort = 1;
  } else if (warp < 8) {
    // ---------------- softmax: one row per thread ----------------
    const int x = warp >> 2;                   // query tile
    const int r = row & 127;
    const uint32_t lane_base = (uint32_t)((warp & 3) * 32) << 16;
    const uint32_t s_col = tmem + lane_base + x * 128;
    const uint32_t o_col = tmem + lane_base + 256 + x * D;
    unsigned char* prow = smem + S::P_OFF + x * S::P_B;
    const float c2 = scale * 1.4426950408889634f;   // scores in log2 units
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
      tc_fence_before();
      mbar_arrive(&s_free[x][bf]);             // the scores are in registers
      const bool full = t0 + kTok - 1 <= pos;  // no key of the tile is masked
      float mx = -INFINITY;
      if (full) {
#pragma unroll
        for (int i = 0; i < kTok; ++i) mx = fmaxf(mx, __uint_as_float(sr[i]));
      } else {
#pragma unroll
        for (int i = 0; i < kTok; ++i)
          if (t0 + i <= pos) mx = fmaxf(mx, __uint_as_float(sr[i]));
      }
      const float m_new = fmaxf(m, mx * c2);   // (c2 > 0: the maximum commutes)
      if (j == 0) {
        m = m_new;
      } else {
        // P(j) overwrites P(j - 1) and a rescale rewrites O: both wait for
        // the MMAs of tile j - 1
        if (!warp_wait(&pv_done[x], (j - 1) & 1, abort)) {
          ok = false;
          break;
        }
        const bool need = m_new > m + kRescale;
        if (__any_sync(0xffffffffu, need)) {
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
          tmem_wait_st();
        }
      }
      float sum = 0.f;
#pragma unroll
      for (int c = 0; c < kTok / 8; ++c) {     // 8 tokens = one 16-byte chunk of P
        float p[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const int i = 8 * c + e;
          const float v = ex2_approx(fmaf(__uint_as_float(sr[i]), c2, -m));
          p[e] = full || t0 + i <= pos ? v : 0.f;
          sum += p[e];
        }
        *reinterpret_cast<uint4*>(prow + sw128(r, c)) =
            make_uint4(pack_h2(p[0], p[1]), pack_h2(p[2], p[3]), pack_h2(p[4], p[5]),
                       pack_h2(p[6], p[7]));
      }
      l += sum;
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      tc_fence_before();
      mbar_arrive(&p_full[x]);
    }
    // ---------------- epilogue ----------------
    if (ok && ntiles > 0 && !warp_wait(&pv_done[x], (ntiles - 1) & 1, abort)) ok = false;
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
                                       M256Layout<D>::ALLOC);
  if (e != cudaSuccess) return e;
  const int nq = kRowsCta / (g.Hq / g.H);
  dim3 grid((L + nq - 1) / nq, g.H, g.B);
  launch_pdl(kern, dim3(grid), dim3(kThreads), (size_t)M256Layout<D>::ALLOC, s, g,
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
// codes, G = 32 (KIVI: 32-token key blocks), head_dim 128, GQA group <= 256.
bool prefill_m256_supported(const Geom& g) {
  const bool fmt_ok = g.fmt == KVQ_FMT_AFFINE || g.fmt == KVQ_FMT_SYMMETRIC || g.fmt == KVQ_FMT_KIVI;
  return fmt_ok && g.act == KVQ_BF16 && g.D == 128 && g.G == 32 && g.kb == g.vb &&
         (g.kb == 2 || g.kb == 4) && g.Hq / g.H <= kRowsCta;
}

cudaError_t launch_prefill_m256(const Geom& g, const void* q, int L, float scale, void* out,
                                int* err, cudaStream_t s) {
  if (g.D == 64) return launch_m256_d<64>(g, q, L, scale, out, err, s);
  return launch_m256_d<128>(g, q, L, scale, out, err, s);
}

}  // namespace kvq
