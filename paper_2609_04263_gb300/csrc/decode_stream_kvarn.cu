// Streaming decode attention over the coded tokens of a KVarN cache, on
// tensor cores in the Hadamard-rotated basis (§3.1 KVarN: coded token t is
// stored as r_t c_j (s_tg code_tj + m_tg) with row scale r_t, per-block column
// scale c_j and per-token group scale/offset; §3.2-3.3 attention over the
// stored reconstruction, L = 1).
//
// The work split, the ring and the merges follow decode_stream.cu: persistent
// CTAs stream equal shares of the flattened (sequence, kv head, 32-token
// block) space of coded blocks; a producer warp copies runs of blocks (codes,
// group metadata, row scales) and each block's column-scale rows into ring
// stages; eight consumer warps take the blocks in turn, tokens as the MMA rows
// and the GQA heads as its columns.
//   scores  q_rot = H q / sqrt(D) (times the softmax scale in log2 units) is
//     formed once per head; per block B = q_rot * c_k as bf16 high + low parts
//     and A = key codes as exact bf16 integers 128 + c, one accumulator per
//     quantization group; the 128 is removed with an MMA over a constant
//     operand (which also gives sum_j q'_j, the offset's weight), then
//       S = r_t sum_g [s_tg (acc_g - bias_g) + m_tg bias_g / 128].
//   values  A = c_v,j * code (fp16), B = fp16(p) * (r_t s_tg); the offsets
//     r_t m_tg enter through a small MMA (rows = groups) and are scaled by
//     c_v,j when the block's contribution is added.
// The sinks and the staged tokens (full precision, original basis) are left
// to attend_kvarn_decode_kernel; this kernel leaves each head's result as one
// more split partial (m, l, o rotated back) in workspace slot kFinalSlot,
// which that kernel (launched next) merges with its own partials.
#include "decode_attn.cuh"
#include "stream_common.cuh"

namespace kvq {
namespace {
using namespace dattn;
using namespace stream;

template <int D, int KB, int VB, int G>
struct KCfg {
  static constexpr int NG32 = D / 32;                 // 32-channel sub-groups (two k-steps each)
  static constexpr int NGG = D / G;                   // quantization groups per token
  static constexpr int MT = D / 16;                   // P V m-tiles
  static constexpr int KCB = D * KB / 8, VCB = D * VB / 8;
  static constexpr int MB = kBT * NGG * 2;            // one group-metadata plane of a block
  // a stage holds kSB consecutive blocks; each plane is contiguous over them
  static constexpr int KC = 0;
  static constexpr int VC = KC + kSB * kBT * KCB;
  static constexpr int KS = VC + kSB * kBT * VCB;
  static constexpr int KZ = KS + kSB * MB;
  static constexpr int VS = KZ + kSB * MB;
  static constexpr int VZ = VS + kSB * MB;
  static constexpr int KR = VZ + kSB * MB;            // row scales, 2 bytes per token
  static constexpr int VR = KR + kSB * kBT * 2;
  static constexpr int KCOL = VR + kSB * kBT * 2;     // one column-scale row per block
  static constexpr int VCOL = KCOL + kSB * D * 2;
  static constexpr int STAGE = (VCOL + kSB * D * 2 + 127) / 128 * 128;
  static_assert(G % kBT == 0 && G % 32 == 0, "blocks lie inside one column-scale block");
  static_assert(NGG <= 8, "offset MMA rows hold the groups");
};

// Normalised Hadamard transform of a row held as x[i] = row[lane + 32 i]
// (butterflies over the lanes, then over the slots, then 1 / sqrt(D)).
template <int D>
__device__ __forceinline__ void fwht_rows(float (&x)[D / 32], int lane, float inv_sqrt_d) {
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

template <int D, int KB, int VB, int G>
__global__ void __launch_bounds__(kThreads, 1)
decode_stream_kvarn_kernel(Geom g, const __nv_bfloat16* __restrict__ q, float scale,
                           float inv_sqrt_d, int* err, int ns) {
  using C = KCfg<D, KB, VB, G>;
  constexpr int NG32 = C::NG32, NGG = C::NGG, MT = C::MT;
  extern __shared__ __align__(128) unsigned char smem[];
  pdl_wait();
  pdl_trigger();

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gid = lane >> 2, tid = lane & 3;
  const int grp = g.Hq / g.H;
  const int PW = grp * (D + 2);
  float* slot = reinterpret_cast<float*>(smem + (size_t)ns * C::STAGE);   // [kNW][PW]
  float* qr = slot + kNW * PW;                       // [8][D] rotated queries, then merged rows
  Merge* mg = reinterpret_cast<Merge*>(qr + 8 * D);
  uint64_t* full = reinterpret_cast<uint64_t*>(mg + 1);
  uint64_t* empty = full + ns;
  float* wsb = reinterpret_cast<float*>(g.pl[KVQ_PLANE_WORKSPACE].p);

  const int T = cache_tokens(g);
  const int S = g.S;
  const int nbq = kvarn_nblocks(T, S, G) * G;        // coded tokens per head
  const int BH = g.B * g.H;
  const int nb = nbq / kBT;                          // blocks per head
  const int64_t N = (int64_t)BH * nb;
  if (N == 0) {                                      // nothing coded: an empty partial
    if (blockIdx.x == 0)
      for (int i = threadIdx.x; i < g.B * g.Hq; i += blockDim.x) {
        float* w = wsb + ((int64_t)i * kMaxSplits + kFinalSlot) * (D + kWsStride);
        w[0] = -INFINITY;
        w[1] = 0.f;
      }
    return;
  }
  const int P = N < (int64_t)gridDim.x ? (int)N : (int)gridDim.x;
  if ((int)blockIdx.x >= P) return;
  const int64_t k0 = range_start(blockIdx.x, N, P), k1 = range_start(blockIdx.x + 1, N, P);
  const int nblk = (int)(k1 - k0);

  if (threadIdx.x == 0) {
    for (int i = 0; i < ns; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], kSB);                     // one arrival per block
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();

  // ------------------------------------------------------------------ producer
  if (warp == kNW) {
    const int nst = (nblk + kSB - 1) / kSB;
    int head = (int)(k0 / nb), blk = (int)(k0 % nb);  // first block of the next stage
    int s = 0;
    for (; s < nst; ++s) {
      const int st = s % ns;
      bool ok = true;
      if (s >= ns && lane == 0) ok = mbar_wait(&empty[st], ((s / ns) - 1) & 1);
      if (!__shfl_sync(0xffffffffu, ok, 0)) {
        if (lane == 0) atomicOr(err, 1);
        break;
      }
      const int nbs = min(kSB, nblk - s * kSB);
      const int h_st = head, b_st = blk;
      unsigned char* sp = smem + (size_t)st * C::STAGE;
      if (lane == 0)
        mbar_expect_tx(&full[st], (uint32_t)nbs * (kBT * (C::KCB + C::VCB) + 4 * C::MB +
                                                   2 * kBT * 2 + 2 * D * 2));
      __syncwarp();
      // runs of one head's blocks: in pass p, lane 8 r + c issues copy c of
      // run 4 p + r (every lane walks the same blocks)
      int nrun = 0;
      for (int pass = 0; pass == 0 || pass * 4 < nrun; ++pass) {
        const int myr = pass * 4 + lane / 8, myc = lane % 8;
        int hh = h_st, bb = b_st, cnt = 0, r_head = 0, r_blk = 0, r_n = 0, r_sub = 0, p_head = -1;
#pragma unroll
        for (int i = 0; i < kSB; ++i) {
          if (i < nbs) {
            if (hh != p_head) {
              if (cnt == myr) { r_head = hh; r_blk = bb; r_sub = i; }
              ++cnt;
              p_head = hh;
            }
            if (cnt - 1 == myr) ++r_n;
            if (++bb == nb) { bb = 0; ++hh; }
          }
        }
        if (pass == 0) {
          nrun = cnt;
          head = hh;
          blk = bb;
        }
        if (myr < nrun) {
          const int qi = r_blk * kBT, nt = r_n * kBT;   // coded-token rows of the run
          const uint8_t* src;
          unsigned char* dst;
          uint32_t bytes;
          const int planes[8] = {KVQ_PLANE_K_CODES, KVQ_PLANE_V_CODES, KVQ_PLANE_K_SCALE,
                                 KVQ_PLANE_K_ZERO, KVQ_PLANE_V_SCALE, KVQ_PLANE_V_ZERO,
                                 KVQ_PLANE_K_ROW, KVQ_PLANE_V_ROW};
          if (myc < 2) {
            src = plane_ptr<uint8_t>(g, planes[myc], 0, r_head, qi);
            dst = sp + (myc == 0 ? C::KC + r_sub * kBT * C::KCB : C::VC + r_sub * kBT * C::VCB);
            bytes = nt * (myc == 0 ? C::KCB : C::VCB);
          } else if (myc < 6) {
            src = reinterpret_cast<const uint8_t*>(plane_ptr<__half>(g, planes[myc], 0, r_head, qi));
            dst = sp + C::KS + (myc - 2) * kSB * C::MB + r_sub * C::MB;
            bytes = r_n * C::MB;
          } else {                                     // row scales: plane row 0, column qi
            src = reinterpret_cast<const uint8_t*>(plane_ptr<__half>(g, planes[myc], 0, r_head, 0, qi));
            dst = sp + (myc == 6 ? C::KR : C::VR) + r_sub * kBT * 2;
            bytes = nt * 2;
          }
          bulk_g2s(dst, src, bytes, &full[st]);
        }
      }
      // each block's column-scale rows (key, value)
      if (lane < 2 * nbs) {
        const int i = lane >> 1, which = lane & 1;
        int hh = h_st, bb = b_st;
#pragma unroll
        for (int j = 0; j < kSB; ++j)
          if (j < i && ++bb == nb) { bb = 0; ++hh; }
        const int crow = bb * kBT / G;
        bulk_g2s(sp + (which ? C::VCOL : C::KCOL) + i * D * 2,
                 plane_ptr<__half>(g, which ? KVQ_PLANE_V_COL : KVQ_PLANE_K_COL, 0, hh, crow),
                 D * 2, &full[st]);
      }
    }
    if (lane == 0)                                   // the last copies land before the CTA ends
      for (int i = max(0, s - ns); i < s; ++i)
        if (!mbar_wait(&full[i % ns], (i / ns) & 1)) atomicOr(err, 1);
    return;
  }

  // ------------------------------------------------------------------ consumers
  const float c2 = scale * 1.4426950408889634f;      // scores in log2 units
  const uint32_t kmask = KB == 4 ? 0x000F000Fu : 0x00030003u;
  const uint32_t vmask = VB == 4 ? 0x000F000Fu : 0x00030003u;
  const __half h1024 = __float2half(1024.f);
  const __half2 bias2 = __halves2half2(h1024, h1024);
  const uint32_t a128[4] = {kMagic, kMagic, kMagic, kMagic};
  const int tc = threadIdx.x;

  float m_run[2], l_run[2];
  float o[MT][4];
  bool bad = false;

  auto process = [&](const unsigned char* sp, int sub) {
    const unsigned char* kc = sp + C::KC + sub * kBT * C::KCB;
    const unsigned char* vc = sp + C::VC + sub * kBT * C::VCB;
    const __half* ks = reinterpret_cast<const __half*>(sp + C::KS + sub * C::MB);
    const __half* kz = reinterpret_cast<const __half*>(sp + C::KZ + sub * C::MB);
    const uint32_t* vs = reinterpret_cast<const uint32_t*>(sp + C::VS + sub * C::MB);
    const uint32_t* vz = reinterpret_cast<const uint32_t*>(sp + C::VZ + sub * C::MB);
    const __half* kr = reinterpret_cast<const __half*>(sp + C::KR + sub * kBT * 2);
    const uint16_t* vr = reinterpret_cast<const uint16_t*>(sp + C::VR + sub * kBT * 2);
    const __half* kcol = reinterpret_cast<const __half*>(sp + C::KCOL + sub * D * 2);
    const __half* vcol = reinterpret_cast<const __half*>(sp + C::VCOL + sub * D * 2);

    // ---------------------------------------------------------------- scores
    float acc[NGG][2][4], bias[NGG][4];
#pragma unroll
    for (int gg = 0; gg < NGG; ++gg) {
      bias[gg][0] = bias[gg][1] = bias[gg][2] = bias[gg][3] = 0.f;
#pragma unroll
      for (int mt = 0; mt < 2; ++mt) acc[gg][mt][0] = acc[gg][mt][1] = acc[gg][mt][2] = acc[gg][mt][3] = 0.f;
    }
#pragma unroll
    for (int gq = 0; gq < NG32; ++gq) {
      const int gg = gq * 32 / G;
      // q' = q_rot * c_k for head gid, channels 32 gq + 8 tid + e
      const float4 qa = *reinterpret_cast<const float4*>(qr + gid * D + 32 * gq + 8 * tid);
      const float4 qb4 = *reinterpret_cast<const float4*>(qr + gid * D + 32 * gq + 8 * tid + 4);
      const uint4 cu = *reinterpret_cast<const uint4*>(kcol + 32 * gq + 8 * tid);
      const __half* ch = reinterpret_cast<const __half*>(&cu);
      float x[8] = {qa.x, qa.y, qa.z, qa.w, qb4.x, qb4.y, qb4.z, qb4.w};
#pragma unroll
      for (int e = 0; e < 8; ++e) x[e] *= __half2float(ch[e]);
      uint32_t qh[2][2], ql[2][2];
#pragma unroll
      for (int sb = 0; sb < 2; ++sb)
#pragma unroll
        for (int hf = 0; hf < 2; ++hf) {
          const int e0 = qk_chan<KB>(sb, hf, 0), e1 = qk_chan<KB>(sb, hf, 1);
          const uint32_t hw = pack_bf16(x[e0], x[e1]);
          const float2 hv = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&hw));
          qh[sb][hf] = hw;
          ql[sb][hf] = pack_bf16(x[e0] - hv.x, x[e1] - hv.y);
        }
#pragma unroll
      for (int sb = 0; sb < 2; ++sb) {
        mma16816(bias[gg], a128, qh[sb][0], qh[sb][1]);
        mma16816(bias[gg], a128, ql[sb][0], ql[sb][1]);
      }
#pragma unroll
      for (int mt = 0; mt < 2; ++mt) {
        const unsigned char* r0 = kc + (16 * mt + gid) * C::KCB;
        const unsigned char* r1 = r0 + 8 * C::KCB;
        uint32_t w0, w1;
        if (KB == 4) {
          w0 = *reinterpret_cast<const uint32_t*>(r0 + 16 * gq + 4 * tid);
          w1 = *reinterpret_cast<const uint32_t*>(r1 + 16 * gq + 4 * tid);
        } else {
          const uint32_t v0 = *reinterpret_cast<const uint16_t*>(r0 + 8 * gq + 2 * tid);
          const uint32_t v1 = *reinterpret_cast<const uint16_t*>(r1 + 8 * gq + 2 * tid);
          w0 = v0 | (v0 << 14);
          w1 = v1 | (v1 << 14);
        }
#pragma unroll
        for (int sb = 0; sb < 2; ++sb) {
          uint32_t a[4];
          a[0] = magic2(w0 >> (8 * sb), kmask);
          a[1] = magic2(w1 >> (8 * sb), kmask);
          a[2] = magic2(w0 >> (8 * sb + 4), kmask);
          a[3] = magic2(w1 >> (8 * sb + 4), kmask);
          mma16816(acc[gg][mt], a, qh[sb][0], qh[sb][1]);
          mma16816(acc[gg][mt], a, ql[sb][0], ql[sb][1]);
        }
      }
    }
    float S[2][4];
#pragma unroll
    for (int mt = 0; mt < 2; ++mt)
#pragma unroll
      for (int r = 0; r < 2; ++r) {
        const int t = 16 * mt + gid + 8 * r;
        float s0 = 0.f, s1 = 0.f;
#pragma unroll
        for (int gg = 0; gg < NGG; ++gg) {
          const float sc = __half2float(ks[t * NGG + gg]), mz = __half2float(kz[t * NGG + gg]);
          s0 += sc * (acc[gg][mt][2 * r] - bias[gg][0]) + mz * bias[gg][0] * (1.f / 128.f);
          s1 += sc * (acc[gg][mt][2 * r + 1] - bias[gg][1]) + mz * bias[gg][1] * (1.f / 128.f);
        }
        const float rt = __half2float(kr[t]);
        S[mt][2 * r] = rt * s0;
        S[mt][2 * r + 1] = rt * s1;
      }

    // --------------------------------------------------------------- softmax
    float mx[2];
#pragma unroll
    for (int jh = 0; jh < 2; ++jh) {
      mx[jh] = fmaxf(fmaxf(S[0][jh], S[0][2 + jh]), fmaxf(S[1][jh], S[1][2 + jh]));
      mx[jh] = fmaxf(mx[jh], __shfl_xor_sync(0xffffffffu, mx[jh], 4));
      mx[jh] = fmaxf(mx[jh], __shfl_xor_sync(0xffffffffu, mx[jh], 8));
      mx[jh] = fmaxf(mx[jh], __shfl_xor_sync(0xffffffffu, mx[jh], 16));
    }
    float alpha[2];
#pragma unroll
    for (int jh = 0; jh < 2; ++jh) {
      const float mn = fmaxf(m_run[jh], mx[jh]);
      alpha[jh] = m_run[jh] == -INFINITY ? 0.f : exp2f(m_run[jh] - mn);
      m_run[jh] = mn;
      l_run[jh] *= alpha[jh];
    }
    if (__any_sync(0xffffffffu, alpha[0] != 1.f || alpha[1] != 1.f)) {
#pragma unroll
      for (int i = 0; i < MT; ++i) {
        o[i][0] *= alpha[0]; o[i][1] *= alpha[1];
        o[i][2] *= alpha[0]; o[i][3] *= alpha[1];
      }
    }
    uint32_t pb[2][2];
#pragma unroll
    for (int mt = 0; mt < 2; ++mt) {
      float p[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        p[i] = exp2f(S[mt][i] - m_run[i & 1]);
        l_run[i & 1] += p[i];
      }
      pb[mt][0] = movmatrix_t(pack_f16(p[0], p[1]));
      pb[mt][1] = movmatrix_t(pack_f16(p[2], p[3]));
    }

    // ------------------------------------------------------------------- P V
    float offb[4] = {0.f, 0.f, 0.f, 0.f};            // sum_t p r_t m_tg, rows = groups
#pragma unroll
    for (int mt = 0; mt < 2; ++mt) {
      int tk[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) tk[i] = 16 * mt + 2 * tid + (i & 1) + 8 * (i >> 1);
      const uint32_t vr01 = (uint32_t)vr[tk[0]] | ((uint32_t)vr[tk[1]] << 16);
      const uint32_t vr89 = (uint32_t)vr[tk[2]] | ((uint32_t)vr[tk[3]] << 16);
      uint32_t a_off[4] = {0u, 0u, 0u, 0u};
      if (gid < NGG) {
        const uint16_t* vzh = reinterpret_cast<const uint16_t*>(vz);
        const uint32_t z01 = (uint32_t)vzh[tk[0] * NGG + gid] | ((uint32_t)vzh[tk[1] * NGG + gid] << 16);
        const uint32_t z89 = (uint32_t)vzh[tk[2] * NGG + gid] | ((uint32_t)vzh[tk[3] * NGG + gid] << 16);
        a_off[0] = hmul2u(vr01, z01);
        a_off[2] = hmul2u(vr89, z89);
      }
      mma16816_f16(offb, a_off, pb[mt][0], pb[mt][1]);
      uint32_t bq[NGG][2];                           // B = P (r_t s_tg) per group
#pragma unroll
      for (int gg = 0; gg < NGG; ++gg) {
        const uint16_t* vsh = reinterpret_cast<const uint16_t*>(vs);
        const uint32_t s01 = (uint32_t)vsh[tk[0] * NGG + gg] | ((uint32_t)vsh[tk[1] * NGG + gg] << 16);
        const uint32_t s89 = (uint32_t)vsh[tk[2] * NGG + gg] | ((uint32_t)vsh[tk[3] * NGG + gg] << 16);
        bq[gg][0] = hmul2u(pb[mt][0], hmul2u(vr01, s01));
        bq[gg][1] = hmul2u(pb[mt][1], hmul2u(vr89, s89));
      }
#pragma unroll
      for (int gq = 0; gq < NG32; ++gq) {
        const int gg = gq * 32 / G;
        uint32_t x01, x89;
        if (VB == 4) {
          x01 = (uint32_t)*reinterpret_cast<const uint16_t*>(vc + tk[0] * C::VCB + 16 * gq + 2 * gid) |
                ((uint32_t)*reinterpret_cast<const uint16_t*>(vc + tk[1] * C::VCB + 16 * gq + 2 * gid) << 16);
          x89 = (uint32_t)*reinterpret_cast<const uint16_t*>(vc + tk[2] * C::VCB + 16 * gq + 2 * gid) |
                ((uint32_t)*reinterpret_cast<const uint16_t*>(vc + tk[3] * C::VCB + 16 * gq + 2 * gid) << 16);
        } else {
          x01 = (uint32_t)vc[tk[0] * C::VCB + 8 * gq + gid] | ((uint32_t)vc[tk[1] * C::VCB + 8 * gq + gid] << 16);
          x89 = (uint32_t)vc[tk[2] * C::VCB + 8 * gq + gid] | ((uint32_t)vc[tk[3] * C::VCB + 8 * gq + gid] << 16);
        }
        // column scales of rows 32 gq + 4 gid + j, each as a (c, c) pair
        const uint2 cw = *reinterpret_cast<const uint2*>(vcol + 32 * gq + 4 * gid);
        const uint32_t cd[4] = {__byte_perm(cw.x, 0, 0x1010), __byte_perm(cw.x, 0, 0x3232),
                                __byte_perm(cw.y, 0, 0x1010), __byte_perm(cw.y, 0, 0x3232)};
        constexpr int SH = VB == 4 ? 4 : 2;
#pragma unroll
        for (int u = 0; u < 2; ++u) {
          uint32_t a[4];
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const uint32_t xx = (k & 2) ? x89 : x01;
            const uint32_t mg16 = magic2h(xx >> (2 * SH * u + (k & 1) * SH), vmask);
            __half2 cv2 = __hsub2(*reinterpret_cast<const __half2*>(&mg16), bias2);   // exact codes
            const uint32_t c = *reinterpret_cast<const uint32_t*>(&cv2);
            a[k] = hmul2u(c, cd[2 * u + (k & 1)]);
          }
          mma16816_f16(o[2 * gq + u], a, bq[gg][0], bq[gg][1]);
        }
      }
    }
    // the block's offsets, scaled by the column scale of each output channel
#pragma unroll
    for (int gq = 0; gq < NG32; ++gq) {
      const int gg = gq * 32 / G;
      const float f0 = __shfl_sync(0xffffffffu, offb[0], 4 * gg + tid);
      const float f1 = __shfl_sync(0xffffffffu, offb[1], 4 * gg + tid);
      const uint2 cw = *reinterpret_cast<const uint2*>(vcol + 32 * gq + 4 * gid);
      const __half* cc = reinterpret_cast<const __half*>(&cw);
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const float ca = __half2float(cc[2 * u]), cb = __half2float(cc[2 * u + 1]);
        o[2 * gq + u][0] += ca * f0;
        o[2 * gq + u][1] += ca * f1;
        o[2 * gq + u][2] += cb * f0;
        o[2 * gq + u][3] += cb * f1;
      }
    }
  };

  // write the partial of head rows h < grp (m in log2 units, rotated o) from
  // merged rows in qr: rotate back, natural-log m, to workspace slot kFinalSlot
  auto final_partial = [&](int b, int hkv, const float* Mh, const float* Lh) {
    consumer_sync();
    if (warp < grp) {
      float x[D / 32];
#pragma unroll
      for (int i = 0; i < D / 32; ++i) x[i] = qr[warp * D + lane + 32 * i];
      fwht_rows<D>(x, lane, inv_sqrt_d);
      float* w = wsb + (((int64_t)b * g.Hq + hkv * grp + warp) * kMaxSplits + kFinalSlot) * (D + kWsStride);
#pragma unroll
      for (int i = 0; i < D / 32; ++i) w[2 + lane + 32 * i] = x[i];
      if (lane == 0) {
        w[0] = Mh[warp] == -INFINITY ? -INFINITY : Mh[warp] * 0.6931471805599453f;
        w[1] = Lh[warp];
      }
    }
    consumer_sync();
  };

  const int hfirst = (int)(k0 / nb), hlast = (int)((k1 - 1) / nb);
  for (int hd = hfirst; hd <= hlast; ++hd) {
    const int64_t hs = (int64_t)hd * nb;
    const int a = (int)(max(k0, hs) - k0), e = (int)(min(k1, hs + nb) - k0);
    const int b = hd / g.H, hkv = hd % g.H;
    // rotated queries of the head (times the softmax scale, log2 units):
    // rows 0-7 of qr, zero for the MMA columns beyond the group
    if (warp < 8) {
      float x[D / 32];
      const bool live = warp < grp;
      const __nv_bfloat16* src = q + ((int64_t)b * g.Hq + hkv * grp + (live ? warp : 0)) * D;
#pragma unroll
      for (int i = 0; i < D / 32; ++i) x[i] = live ? __bfloat162float(src[lane + 32 * i]) : 0.f;
      fwht_rows<D>(x, lane, inv_sqrt_d);
#pragma unroll
      for (int i = 0; i < D / 32; ++i) qr[warp * D + lane + 32 * i] = x[i] * c2;
    }
    consumer_sync();
    const int jst = a + ((warp - a) % kNW + kNW) % kNW;
    const bool mine = jst < e;
    m_run[0] = m_run[1] = -INFINITY;
    l_run[0] = l_run[1] = 0.f;
#pragma unroll
    for (int i = 0; i < MT; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
    for (int j = jst; j < e && !bad; j += kNW) {
      const int sj = j / kSB, st = sj % ns;
      bool ok = true;
      if (lane == 0) ok = mbar_wait(&full[st], (sj / ns) & 1);
      if (!__shfl_sync(0xffffffffu, ok, 0)) {
        if (lane == 0) atomicOr(err, 1);
        bad = true;
        break;
      }
      process(smem + (size_t)st * C::STAGE, j % kSB);
      __syncwarp();
      if (lane == 0) mbar_arrive1(&empty[st]);
    }
    if (mine) {
#pragma unroll
      for (int jh = 0; jh < 2; ++jh) {
        l_run[jh] += __shfl_xor_sync(0xffffffffu, l_run[jh], 4);
        l_run[jh] += __shfl_xor_sync(0xffffffffu, l_run[jh], 8);
        l_run[jh] += __shfl_xor_sync(0xffffffffu, l_run[jh], 16);
        if (bad) m_run[jh] = -INFINITY;
      }
    }
    consumer_sync();
    if (mine) {
      float* ws = slot + warp * PW;
#pragma unroll
      for (int i = 0; i < MT; ++i) {
        const int d0 = 32 * (i >> 1) + 4 * gid + 2 * (i & 1);
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          const int h = 2 * tid + (r & 1);
          if (h < grp) ws[h * (D + 2) + 2 + d0 + (r >> 1)] = o[i][r];
        }
      }
      if (gid == 0)
#pragma unroll
        for (int jh = 0; jh < 2; ++jh)
          if (2 * tid + jh < grp) {
            ws[(2 * tid + jh) * (D + 2)] = m_run[jh];
            ws[(2 * tid + jh) * (D + 2) + 1] = l_run[jh];
          }
    }
    consumer_sync();
    const int np = min(kNW, e - a);
    if (tc < grp) {
      float M = -INFINITY;
      for (int i = 0; i < np; ++i) M = fmaxf(M, slot[((a + i) % kNW) * PW + tc * (D + 2)]);
      float L = 0.f;
      for (int i = 0; i < np; ++i) {
        const float* pp = slot + ((a + i) % kNW) * PW + tc * (D + 2);
        const float w = pp[0] == -INFINITY ? 0.f : exp2f(pp[0] - M);
        mg->m[i][tc] = w;
        L += w * pp[1];
      }
      mg->M[tc] = M;
      mg->L[tc] = L;
    }
    consumer_sync();
    const int c0 = cta_of(hs, N, P), c1 = cta_of(hs + nb - 1, N, P);
    const int nct = c1 - c0 + 1;
    if (nct > kMaxSplits - 1) {                      // the host sizes the grid so this cannot happen
      if (tc == 0) atomicOr(err, 4);
      continue;
    }
    const int64_t orow0 = (int64_t)b * g.Hq + hkv * grp;
    for (int idx = tc; idx < grp * D; idx += kNW * 32) {
      const int h = idx / D, d = idx % D;
      float acc = 0.f;
      for (int i = 0; i < np; ++i) acc += mg->m[i][h] * slot[((a + i) % kNW) * PW + h * (D + 2) + 2 + d];
      if (nct == 1) qr[h * D + d] = acc;
      else wsb[((orow0 + h) * kMaxSplits + (blockIdx.x - c0)) * (D + kWsStride) + 2 + d] = acc;
    }
    if (nct == 1) {
      final_partial(b, hkv, mg->M, mg->L);
      continue;
    }
    if (tc < grp) {
      float* wr = wsb + ((orow0 + tc) * kMaxSplits + (blockIdx.x - c0)) * (D + kWsStride);
      wr[0] = mg->M[tc];
      wr[1] = mg->L[tc];
    }
    consumer_sync();
    if (tc == 0) {
      __threadfence();
      mg->last = atomicAdd(&g.counters[hd], 1u) == (unsigned)nct - 1;
    }
    consumer_sync();
    if (!mg->last) continue;
    __threadfence();
    if (tc < grp * nct) {
      const int h = tc / nct, i = tc % nct;
      const float* wr = wsb + ((orow0 + h) * kMaxSplits + i) * (D + kWsStride);
      mg->m[i][h] = __ldcg(wr);
      mg->l[i][h] = __ldcg(wr + 1);
    }
    consumer_sync();
    if (tc < grp) {
      float M = -INFINITY;
      for (int i = 0; i < nct; ++i) M = fmaxf(M, mg->m[i][tc]);
      float L = 0.f;
      for (int i = 0; i < nct; ++i) {
        const float w = mg->m[i][tc] == -INFINITY ? 0.f : exp2f(mg->m[i][tc] - M);
        mg->m[i][tc] = w;
        L += w * mg->l[i][tc];
      }
      mg->M[tc] = M;
      mg->L[tc] = L;
    }
    consumer_sync();
    for (int idx = tc; idx < grp * D; idx += kNW * 32) {
      const int h = idx / D, d = idx % D;
      const float* wr = wsb + (orow0 + h) * kMaxSplits * (D + kWsStride) + 2 + d;
      float acc = 0.f;
#pragma unroll 4
      for (int i = 0; i < nct; ++i) acc += mg->m[i][h] * __ldcg(wr + i * (D + kWsStride));
      qr[h * D + d] = acc;
    }
    if (tc == 0) g.counters[hd] = 0;                 // ready for the next call
    final_partial(b, hkv, mg->M, mg->L);
  }
}

template <int D, int KB, int VB, int G>
size_t stream_smem(int grp, int* ns) {
  using C = KCfg<D, KB, VB, G>;
  const size_t fixed = (size_t)kNW * grp * (D + 2) * 4 + (size_t)8 * D * 4 + sizeof(Merge);
  int n = (int)((kSmemMax - fixed) / (C::STAGE + 16));
  if (n > kMaxStages) n = kMaxStages;
  *ns = n;
  return (size_t)n * C::STAGE + fixed + (size_t)2 * n * 8;
}

template <int D, int KB, int VB, int G>
cudaError_t launch_t(const Geom& g, const void* q, float scale, int* err, cudaStream_t s) {
  const int grp = g.Hq / g.H;
  int ns = 0;
  const size_t sm = stream_smem<D, KB, VB, G>(grp, &ns);
  auto kern = decode_stream_kvarn_kernel<D, KB, VB, G>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
  if (e != cudaSuccess) return e;
  launch_pdl(kern, dim3(decode_stream_ctas(g)), dim3(kThreads), sm, s, g,
             reinterpret_cast<const __nv_bfloat16*>(q), scale, (float)(1.0 / sqrt((double)D)), err, ns);
  return cudaGetLastError();
}

}  // namespace

bool decode_stream_kvarn_supported(const Geom& g) {
  const bool shape = (g.D == 256 && g.G == 64) || (g.D == 64 && g.G == 32);
  return g.fmt == KVQ_FMT_KVARN && g.act == KVQ_BF16 && shape && g.kb == 4 && g.vb == 2 &&
         g.Hq / g.H <= 8;
}

cudaError_t launch_decode_stream_kvarn(const Geom& g, const void* q, float scale, int* err,
                                       cudaStream_t s) {
  if (g.D == 256) return launch_t<256, 4, 2, 64>(g, q, scale, err, s);
  return launch_t<64, 4, 2, 32>(g, q, scale, err, s);
}

}  // namespace kvq
