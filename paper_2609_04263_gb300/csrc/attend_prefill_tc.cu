// Causal GQA prefill attention over the stored reconstruction on the
// 5th-generation tensor cores (tcgen05), Sections 3.1-3.3: the L newest
// queries attend to all tokens up to their own position, and every key and
// value is the cache's reconstruction (codes x scale + offset).
//
// One CTA = 128 query rows (the g query heads of one kv head x 128/g
// consecutive queries) of one sequence; keys and values stream in tiles of
// 128 tokens.  Three roles:
//   producers (warps 4-7): one token per thread; reconstruct K as bf16 high
//     part + bf16 remainder (about 16 significant bits, which large logits
//     need) and V as fp16, into double-buffered shared tiles in the 128-byte
//     swizzled K-major layout of the MMA descriptors (V transposed: d rows,
//     tokens along K);
//   issuer (warp 8, one thread): S = Q K_hi^T + Q K_lo^T into a double-buffered
//     TMEM tile (128 x 128 fp32), and, one tile behind, O_tile = P V into a
//     double-buffered TMEM tile (128 x 64 fp32), each completion signalled by
//     tcgen05.commit on an mbarrier;
//   softmax (warps 0-3): thread r owns row r (TMEM lane r): reads its 128
//     scores, applies the causal mask and the online softmax in log2 units,
//     writes P as fp16 into the swizzled P tile and accumulates
//     O = O alpha + O_tile in registers.
// Every wait is bounded and also gives up when another role has timed out;
// the issuer drains its MMAs before TMEM is freed, and a timed-out CTA
// stores nothing and sets the library's error word.
#include <math.h>

#include "tc_common.cuh"

namespace kvq {
namespace {
using namespace tc;

constexpr int kRows = 128;                 // query rows per CTA (MMA M)
constexpr int kTok = 128;                  // tokens per tile (QK^T N, PV K)
constexpr int kThreads = 288;              // 4 softmax + 4 producer warps + issuer warp

// shared memory (bytes from a 1024-aligned base); D = 64
struct PfLayout {
  static constexpr int Q_OFF = 0;                           // [128 rows][64] bf16, one atom
  static constexpr int KV_OFF = 16384;
  static constexpr int KH = 0, KL = 16384, VT = 32768;     // within a KV buffer
  static constexpr int KV_B = 49152;                        // K hi, K lo, V^T (2 atoms x 64 rows)
  static constexpr int P_OFF = KV_OFF + 2 * KV_B;           // [2 atoms][128 rows][128 B] fp16
  static constexpr int P_B = 32768;
  static constexpr int TOTAL = P_OFF + 2 * P_B;
  static constexpr int ALLOC = TOTAL + 1024;                // alignment slack
};

// Byte offset of 16-byte chunk c of row r in a K-major 128-byte-swizzled
// tile (rows of 128 bytes, 8-row groups 1024 bytes apart).
__device__ __forceinline__ int sw128(int r, int c) {
  return (r >> 3) * 1024 + (r & 7) * 128 + ((c ^ (r & 7)) << 4);
}

// What one producer thread loads per tile (affine/symmetric cache, G = 32,
// D = 64): the K code row of its token with the token's fp16 scales (and
// offsets), and, for its block of V (8 tokens x 8 channels), each token's
// code word of those channels with the scale (and offset) of their group.
template <int BITS>
struct TokenCodes {
  uint4 kc[BITS / 2];                  // D * BITS / 8 bytes
  uint32_t ks, kz;                     // two fp16 per word (groups 0, 1)
  uint32_t vw[8];                      // 8 codes of channels 8dc .. 8dc+7, per token
  __half vs[8], vz[8];
};

template <int BITS, bool SYM>
__device__ __forceinline__ void load_token(const Geom& g, int b, int h, int t, int vt0, int dc,
                                           int T, TokenCodes<BITS>& r) {
  if (t < T) {
    const uint4* kc = reinterpret_cast<const uint4*>(plane_ptr<uint8_t>(g, KVQ_PLANE_K_CODES, b, h, t));
#pragma unroll
    for (int i = 0; i < BITS / 2; ++i) r.kc[i] = __ldg(kc + i);
    r.ks = __ldg(reinterpret_cast<const uint32_t*>(plane_ptr<__half>(g, KVQ_PLANE_K_SCALE, b, h, t)));
    r.kz = SYM ? 0u
               : __ldg(reinterpret_cast<const uint32_t*>(plane_ptr<__half>(g, KVQ_PLANE_K_ZERO, b, h, t)));
  } else {                            // beyond the cache: reconstructs as zeros
#pragma unroll
    for (int i = 0; i < BITS / 2; ++i) r.kc[i] = make_uint4(0, 0, 0, 0);
    r.ks = r.kz = 0;
  }
  const __half hz = __float2half_rn(0.f);
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int tv = vt0 + i;
    if (tv < T) {
      const uint8_t* row = plane_ptr<uint8_t>(g, KVQ_PLANE_V_CODES, b, h, tv);
      r.vw[i] = BITS == 4 ? __ldg(reinterpret_cast<const uint32_t*>(row) + dc)
                          : (uint32_t)__ldg(reinterpret_cast<const unsigned short*>(row) + dc);
      r.vs[i] = __ldg(plane_ptr<__half>(g, KVQ_PLANE_V_SCALE, b, h, tv, dc >> 2));
      r.vz[i] = SYM ? hz : __ldg(plane_ptr<__half>(g, KVQ_PLANE_V_ZERO, b, h, tv, dc >> 2));
    } else {
      r.vw[i] = 0;
      r.vs[i] = r.vz[i] = hz;
    }
  }
}

// Channels 8c .. 8c+7 reconstructed as code x scale + offset (offset
// -2^(b-1) scale for symmetric codes), as the cache's other readers do.
template <int BITS, bool SYM>
__device__ __forceinline__ void recon8(const uint4 (&codes)[BITS / 2], uint32_t sw, uint32_t zw,
                                       int c, float v[8]) {
  const uint32_t* w32 = reinterpret_cast<const uint32_t*>(codes);
  const uint32_t w = BITS == 4 ? w32[c] : (w32[c >> 1] >> (16 * (c & 1))) & 0xFFFFu;
  const int grp = c >> 2;                        // 32-channel group
  const __half2 s2 = *reinterpret_cast<const __half2*>(&sw);
  const __half2 z2 = *reinterpret_cast<const __half2*>(&zw);
  const float s = grp ? __high2float(s2) : __low2float(s2);
  const float m = SYM ? -(float)(1 << (BITS - 1)) * s : (grp ? __high2float(z2) : __low2float(z2));
  constexpr unsigned mask = (1u << BITS) - 1;
#pragma unroll
  for (int e = 0; e < 8; ++e) v[e] = (float)((w >> (e * BITS)) & mask) * s + m;
}

__device__ __forceinline__ uint32_t pack_h2(float lo, float hi) {
  __half2 v = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

template <int BITS, bool SYM>
__global__ void __launch_bounds__(kThreads, 1)
attend_prefill_tc_kernel(Geom g, const __nv_bfloat16* __restrict__ q, int L, float scale,
                         __nv_bfloat16* __restrict__ out, int nq, int* err) {
  pdl_wait();
  pdl_trigger();
  constexpr int D = 64;
  using S = PfLayout;
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ uint64_t kv_full[2], kv_free[2], s_full[2], s_free[2], p_full[2], o_full[2],
      o_free[2], done_bar;
  __shared__ uint32_t tmem_base;
  __shared__ int abort_flag;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nqt = gridDim.x;
  const int qtile = nqt - 1 - blockIdx.x;             // longest first
  const int hkv = blockIdx.y, b = blockIdx.z;
  const int grp = g.Hq / g.H;
  const int T = cache_tokens(g);
  const int tq = g.fmt == KVQ_FMT_KIVI ? kivi_tq(T, g.R, g.G) : T;
  const int q0 = qtile * nq;
  const int nql = min(nq, L - q0);
  const int pos_first = T - L + q0;
  const int t_end = pos_first + nql;                  // keys [0, t_end)
  const int ntiles = (t_end + kTok - 1) / kTok;
  volatile int* abort = &abort_flag;

  if (threadIdx.x == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(&kv_full[i], 128);
      mbar_init(&kv_free[i], 1);
      mbar_init(&s_full[i], 1);
      mbar_init(&s_free[i], 128);
      mbar_init(&p_full[i], 128);
      mbar_init(&o_full[i], 1);
      mbar_init(&o_free[i], 128);
    }
    mbar_init(&done_bar, 1);
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (warp == 8) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 512;"
                 ::"r"(smem_u32(&tmem_base)));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  // queries -> the swizzled Q tile (softmax threads, one row each)
  const int row = threadIdx.x;                        // for the softmax role
  int pos = -1;
  if (warp < 4) {
    const int hl = row / nq, qi = row % nq;
    const bool valid = hl < grp && qi < nql;
    if (valid) pos = pos_first + qi;
    const __nv_bfloat16* src = q + (((int64_t)b * g.Hq + hkv * grp + hl) * L + q0 + qi) * D;
#pragma unroll
    for (int c = 0; c < 8; ++c) {
      uint4 v = make_uint4(0, 0, 0, 0);
      if (valid) v = *reinterpret_cast<const uint4*>(src + 8 * c);
      *reinterpret_cast<uint4*>(smem + S::Q_OFF + sw128(row, c)) = v;
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base;

  if (warp >= 4 && warp < 8) {
    // ---------------- producers: reconstruct K and V tiles ----------------
    const int t = threadIdx.x - 128;                  // K: token t of the tile
    const int dc = t & 7, tb = t >> 3;                // V: channels 8dc.., tokens 8tb..
    TokenCodes<BITS> cur, nxt;
    if (ntiles > 0) load_token<BITS, SYM>(g, b, hkv, t, 8 * tb, dc, T, cur);
    for (int j = 0; j < ntiles; ++j) {
      const int bf = j & 1;
      if (j + 1 < ntiles)
        load_token<BITS, SYM>(g, b, hkv, (j + 1) * kTok + t, (j + 1) * kTok + 8 * tb, dc, T, nxt);
      if (j >= 2 && !mbar_wait_or_abort(&kv_free[bf], ((j - 2) >> 1) & 1, abort)) break;
      unsigned char* kv = smem + S::KV_OFF + bf * S::KV_B;
#pragma unroll
      for (int c = 0; c < 8; ++c) {
        float v[8];
        recon8<BITS, SYM>(cur.kc, cur.ks, cur.kz, c, v);
        uint32_t h[4], l[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const __nv_bfloat162 hb = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
          const float2 hf = __bfloat1622float2(hb);
          h[i] = *reinterpret_cast<const uint32_t*>(&hb);
          const __nv_bfloat162 lb = __floats2bfloat162_rn(v[2 * i] - hf.x, v[2 * i + 1] - hf.y);
          l[i] = *reinterpret_cast<const uint32_t*>(&lb);
        }
        *reinterpret_cast<uint4*>(kv + S::KH + sw128(t, c)) = make_uint4(h[0], h[1], h[2], h[3]);
        *reinterpret_cast<uint4*>(kv + S::KL + sw128(t, c)) = make_uint4(l[0], l[1], l[2], l[3]);
      }
      // V^T block: rows d = 8dc + e, tokens 8tb .. 8tb+7 (one 16-byte chunk each)
      {
        float vv[8][8];                               // [token][channel]
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const float s = __half2float(cur.vs[i]);
          const float m = SYM ? -(float)(1 << (BITS - 1)) * s : __half2float(cur.vz[i]);
          constexpr unsigned mask = (1u << BITS) - 1;
#pragma unroll
          for (int e = 0; e < 8; ++e) vv[i][e] = (float)((cur.vw[i] >> (e * BITS)) & mask) * s + m;
        }
        unsigned char* vt = kv + S::VT + (tb >> 3) * 8192;
#pragma unroll
        for (int e = 0; e < 8; ++e)
          *reinterpret_cast<uint4*>(vt + sw128(8 * dc + e, tb & 7)) =
              make_uint4(pack_h2(vv[0][e], vv[1][e]), pack_h2(vv[2][e], vv[3][e]),
                         pack_h2(vv[4][e], vv[5][e]), pack_h2(vv[6][e], vv[7][e]));
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      mbar_arrive(&kv_full[bf]);
      cur = nxt;
    }
  } else if (warp == 8 && lane == 0) {
    // ---------------- MMA issuer ----------------
    constexpr uint32_t id_qk = idesc_bf16(kRows, kTok);
    constexpr uint32_t id_pv = idesc_f16(kRows, D);
    for (int j = 0; j <= ntiles; ++j) {
      if (j < ntiles) {
        const int bf = j & 1;
        if (!mbar_wait_or_abort(&kv_full[bf], (j >> 1) & 1, abort)) break;
        if (j >= 2 && !mbar_wait_or_abort(&s_free[bf], ((j - 2) >> 1) & 1, abort)) break;
        tc_fence_after();
        const unsigned char* kv = smem + S::KV_OFF + bf * S::KV_B;
        const uint32_t ts = tmem + bf * kTok;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint64_t qd = sw128_desc(smem + S::Q_OFF + kk * 32);
          umma(ts, qd, sw128_desc(kv + S::KH + kk * 32), id_qk, kk > 0);
          umma(ts, qd, sw128_desc(kv + S::KL + kk * 32), id_qk, 1);
        }
        umma_commit(&s_full[bf]);
      }
      if (j >= 1) {
        const int jj = j - 1, bf = jj & 1;
        if (!mbar_wait_or_abort(&p_full[bf], (jj >> 1) & 1, abort)) break;
        if (jj >= 2 && !mbar_wait_or_abort(&o_free[bf], ((jj - 2) >> 1) & 1, abort)) break;
        tc_fence_after();
        const unsigned char* kv = smem + S::KV_OFF + bf * S::KV_B;
        const unsigned char* p = smem + S::P_OFF + bf * S::P_B;
        const uint32_t to = tmem + 2 * kTok + bf * D;
#pragma unroll
        for (int kk = 0; kk < kTok / 16; ++kk) {
          const int a = kk >> 2, k4 = (kk & 3) * 32;
          umma(to, sw128_desc(p + a * 16384 + k4), sw128_desc(kv + S::VT + a * 8192 + k4), id_pv,
               kk > 0);
        }
        umma_commit(&o_full[bf]);
        umma_commit(&kv_free[bf]);
      }
    }
    umma_commit(&done_bar);                    // every MMA issued above has completed
    if (!mbar_wait(&done_bar, 0)) *abort = 1;
  } else if (warp < 4) {
    // ---------------- softmax: one row per thread ----------------
    const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
    const float c2 = scale * 1.4426950408889634f;  // scores in log2 units
    float m = -INFINITY, l = 0.f, alpha_prev = 1.f;
    float o[D];
#pragma unroll
    for (int i = 0; i < D; ++i) o[i] = 0.f;
    bool ok = true;
    float alpha = 1.f;
    // iteration j: the scores of tile j (j < ntiles), then O += tile j - 1
    for (int j = 0; j <= ntiles && ok; ++j) {
      if (j < ntiles) {
        const int bf = j & 1, t0 = j * kTok;
        if (!mbar_wait_or_abort(&s_full[bf], (j >> 1) & 1, abort)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const bool full = t0 + kTok - 1 <= pos;         // no key of the tile is masked
        // two passes over the scores in TMEM: the row max, then exp2 and P
        const uint32_t srow = tmem + lane_base + bf * kTok;
        float mx = -INFINITY;
#pragma unroll 1
        for (int c0 = 0; c0 < kTok; c0 += 32) {
          uint32_t sr[32];
          tmem_ld16_nowait(srow + c0, sr);
          tmem_ld16_nowait(srow + c0 + 16, sr + 16);
          tmem_wait_ld();
          if (full) {
#pragma unroll
            for (int i = 0; i < 32; ++i) mx = fmaxf(mx, __uint_as_float(sr[i]));
          } else {
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if (t0 + c0 + i <= pos) mx = fmaxf(mx, __uint_as_float(sr[i]));
          }
        }
        mx *= c2;                                      // (c2 > 0: the max commutes)
        const float m_new = fmaxf(m, mx);
        alpha = m_new == -INFINITY ? 1.f : exp2f(m - m_new);
        float sum = 0.f;
        unsigned char* prow = smem + S::P_OFF + bf * S::P_B;
#pragma unroll 1
        for (int c0 = 0; c0 < kTok; c0 += 32) {
          uint32_t sr[32];
          tmem_ld16_nowait(srow + c0, sr);
          tmem_ld16_nowait(srow + c0 + 16, sr + 16);
          tmem_wait_ld();
#pragma unroll
          for (int c = 0; c < 4; ++c) {               // 8 tokens = one 16-byte chunk of P
            float p[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              const int i = 8 * c + e;
              const float x = exp2f(fmaf(__uint_as_float(sr[i]), c2, -m_new));
              p[e] = full || t0 + c0 + i <= pos ? x : 0.f;
              sum += p[e];
            }
            const int ch = (c0 >> 3) + c;               // chunk 0..15 along the tile
            *reinterpret_cast<uint4*>(prow + (ch >> 3) * 16384 + sw128(row, ch & 7)) =
                make_uint4(pack_h2(p[0], p[1]), pack_h2(p[2], p[3]), pack_h2(p[4], p[5]),
                           pack_h2(p[6], p[7]));
          }
        }
        tc_fence_before();
        mbar_arrive(&s_free[bf]);
        l = l * alpha + sum;
        m = m_new;
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        mbar_arrive(&p_full[bf]);
      }
      if (j >= 1) {                                   // O = O alpha(j - 1) + O_tile(j - 1)
        const int jj = j - 1, bf = jj & 1;
        if (!mbar_wait_or_abort(&o_full[bf], (jj >> 1) & 1, abort)) {
          ok = false;
          break;
        }
        tc_fence_after();
#pragma unroll
        for (int c = 0; c < D; c += 16) {
          uint32_t r[16];
          tmem_ld16_nowait(tmem + lane_base + 2 * kTok + bf * D + c, r);
          tmem_wait_ld();
#pragma unroll
          for (int i = 0; i < 16; ++i) o[c + i] = o[c + i] * alpha_prev + __uint_as_float(r[i]);
        }
        tc_fence_before();
        mbar_arrive(&o_free[bf]);
      }
      alpha_prev = alpha;
    }
    // ---------------- epilogue ----------------
    if (ok && !*abort && pos >= 0) {
      const int hl = row / nq, qi = row % nq;
      const float inv = l > 0.f ? 1.f / l : 0.f;
      __nv_bfloat16* dst = out + (((int64_t)b * g.Hq + hkv * grp + hl) * L + q0 + qi) * D;
#pragma unroll
      for (int c = 0; c < 8; ++c) {
        uint32_t w[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const __nv_bfloat162 v = __floats2bfloat162_rn(o[8 * c + 2 * i] * inv,
                                                         o[8 * c + 2 * i + 1] * inv);
          w[i] = *reinterpret_cast<const uint32_t*>(&v);
        }
        *reinterpret_cast<uint4*>(dst + 8 * c) = make_uint4(w[0], w[1], w[2], w[3]);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0 && *abort) atomicOr(err, 8);
  if (warp == 8) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 512;" ::"r"(tmem));
  }
}

}  // namespace

// bf16 affine/symmetric caches with 2/4-bit codes, G = 32, head_dim 64.
bool prefill_tc_supported(const Geom& g) {
  const bool fmt_ok = g.fmt == KVQ_FMT_AFFINE || g.fmt == KVQ_FMT_SYMMETRIC;
  return fmt_ok && g.act == KVQ_BF16 && g.D == 64 && g.G == 32 && g.kb == g.vb &&
         (g.kb == 2 || g.kb == 4) && g.Hq / g.H <= kRows;
}

cudaError_t launch_prefill_tc(const Geom& g, const void* q, int L, float scale, void* out,
                              int* err, cudaStream_t s) {
  const int grp = g.Hq / g.H;
  const int nq = kRows / grp;
  const bool sym = g.fmt == KVQ_FMT_SYMMETRIC;
  auto kern = g.kb == 4 ? (sym ? attend_prefill_tc_kernel<4, true> : attend_prefill_tc_kernel<4, false>)
                        : (sym ? attend_prefill_tc_kernel<2, true> : attend_prefill_tc_kernel<2, false>);
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       PfLayout::ALLOC);
  if (e != cudaSuccess) return e;
  dim3 grid((L + nq - 1) / nq, g.H, g.B);
  launch_pdl(kern, dim3(grid), dim3(kThreads), (size_t)PfLayout::ALLOC, s, g,
             reinterpret_cast<const __nv_bfloat16*>(q), L, scale,
             reinterpret_cast<__nv_bfloat16*>(out), nq, err);
  return cudaGetLastError();
}

}  // namespace kvq
