// LoRA-adapted Q/K/V projection on the 5th-generation tensor cores (tcgen05),
// for many rows (prefill).  Section 3, Eq. (1) and Eq. (lora), with the
// adapter kept as an explicit rank-r branch (Section 3.4):
//   y = x W_p^T + (alpha/r) (x A_p^T) B_p^T,   then RoPE on q and k.
//
// One CTA computes a 128 x BN tile of y inside one projection p (BN holds
// whole heads).  Thread 0 streams K-slices of x, W and A_p with TMA
// (128-byte swizzle) through a kStages-deep mbarrier ring; thread 32 issues
// tcgen05.mma: x W^T accumulates in TMEM columns [0, BN), x A_p^T in columns
// [BN, BN + RP).  Afterwards the 128 threads (one per row / TMEM lane) read
// x A_p^T, scale it by alpha/r, round it to bf16 and write it to shared
// memory as an MMA operand; one more MMA pass adds (alpha/r)(x A_p^T) B_p^T
// into the main accumulator.  The epilogue reads the tile from TMEM, applies
// rotate-half RoPE and stores head-major [B, H, L, D].  Every mbarrier wait is
// bounded; a timeout sets the library's error word and the CTA still frees
// its TMEM.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <math.h>
#include <string.h>

#include <mutex>

#include "kvq_internal.cuh"
#include "quant_common.cuh"
#include "tc_common.cuh"

namespace kvq {

// shared with project.cu
void rope_theta_table(float rope_base, int D, float* hi, float* lo);

namespace {

constexpr int BM = 128;
constexpr int BK = 64;              // bf16 elements per 128-byte swizzle row
constexpr int kStages = 3;
constexpr int kThreads = 128;      // + 256 dequantising threads over an NF4 base
constexpr int kDqWarps = 8;
using namespace tc;

// The 16 NF4 levels, code 0 .. 15, as QLoRA publishes the data type.
__constant__ float c_nf4_lv[16] = {
    -1.0f, -0.6961928009986877f, -0.5250730514526367f, -0.39491748809814453f,
    -0.28444138169288635f, -0.18477343022823334f, -0.09105003625154495f, 0.0f,
    0.07958029955625534f, 0.16093020141124725f, 0.24611230194568634f, 0.33791524171829224f,
    0.44070982933044434f, 0.5626170039176941f, 0.7229568362236023f, 1.0f};

struct TcArgs {
  void* out[3];
  int B, L, M, D, Hq, Hkv;
  int n_off[4];                 // first output column of q, k, v; total columns
  int r[3], rp[3];              // ranks and ranks padded to 16
  int pos0;
  const int* pos_dev;
  int pos_stride;
  float alpha_over_r;
  int rope;
  int k_blocks;
  int* err;
  int pack;                     // 1: code k and v into the cache g instead of storing them
  const uint8_t* nf4_codes;     // NF4 base: codes [N][d_in / 2] (two inputs a byte, low first)
  const float* nf4_absmax;      //           and one absmax per 64 inputs of a row [N][d_in / 64]
  float* plain_out;             // plain product: fp32 [M][N] row-major, no RoPE, no adapters
  int kb_wrap;                  // > 0: K slice kb of W is slice kb % kb_wrap (W repeated along K)
  Geom g;
  float theta_hi[128], theta_lo[128];
};

__device__ __forceinline__ void rope_cs(int pos, float th_hi, float th_lo, float* c, float* s) {
  const float x = (float)pos;
  const float p = x * th_hi;
  const float e = fmaf(x, th_hi, -p) + x * th_lo;
  const float k = rintf(p * 0.15915494309189535f);
  float r = fmaf(-k, 6.28125f, p);
  r = fmaf(-k, 1.9353071795864769e-3f, r);
  r = fmaf(-k, 1.0253132e-11f, r);
  r += e;
  sincosf(r, s, c);
}

// Rotate-half pair (a, b) by the angle with cosine c and sine s.  Products
// are rounded before the fused add, so both epilogues (bf16 store, or coding
// into the cache) produce the same values bit for bit.
__device__ __forceinline__ void rope_rot(float& a, float& b, float c, float s) {
  const float a0 = a, b0 = b;
  a = fmaf(a0, c, -__fmul_rn(b0, s));
  b = fmaf(b0, c, __fmul_rn(a0, s));
}

// One token's group of 32 channels (values already rounded to bf16, as the
// unfused path stores them) coded into the cache planes: 4 x 8 codes LSB
// first, fp16 scale (and offset).
template <int BITS, bool SYM>
__device__ __forceinline__ void code_group32(const Geom& g, int cplane, int splane, int zplane,
                                             int b, int h, int t, int gi, const float v[32]) {
  float lo = v[0], hi = SYM ? fabsf(v[0]) : v[0];
#pragma unroll
  for (int i = 1; i < 32; ++i) {
    if (SYM) hi = fmaxf(hi, fabsf(v[i]));
    else { lo = fminf(lo, v[i]); hi = fmaxf(hi, v[i]); }
  }
  uint64_t w[4];
  float s = 0.f;
#pragma unroll
  for (int q = 0; q < 4; ++q) w[q] = quant::code8<BITS, SYM>(v + 8 * q, lo, hi, &s);
  uint8_t* crow = plane_ptr<uint8_t>(g, cplane, b, h, t) + gi * (32 * BITS / 8);
  if (BITS == 2) {
    *reinterpret_cast<uint2*>(crow) = make_uint2((uint32_t)w[0] | ((uint32_t)w[1] << 16),
                                                 (uint32_t)w[2] | ((uint32_t)w[3] << 16));
  } else if (BITS == 4) {
    *reinterpret_cast<uint4*>(crow) =
        make_uint4((uint32_t)w[0], (uint32_t)w[1], (uint32_t)w[2], (uint32_t)w[3]);
  } else {
    uint4* d = reinterpret_cast<uint4*>(crow);
    d[0] = make_uint4((uint32_t)w[0], (uint32_t)(w[0] >> 32), (uint32_t)w[1], (uint32_t)(w[1] >> 32));
    d[1] = make_uint4((uint32_t)w[2], (uint32_t)(w[2] >> 32), (uint32_t)w[3], (uint32_t)(w[3] >> 32));
  }
  *plane_ptr<__half>(g, splane, b, h, t, gi) = __float2half_rn(s);
  if (!SYM) *plane_ptr<__half>(g, zplane, b, h, t, gi) = __float2half_rn(lo + 0.0f);
}

template <int BITS, bool SYM>
__device__ __forceinline__ void code_pair(const Geom& g, int which, int b, int h, int t, int g1,
                                          int g2, const float* x1, const float* x2) {
  const int cp = which ? KVQ_PLANE_V_CODES : KVQ_PLANE_K_CODES;
  const int sp = which ? KVQ_PLANE_V_SCALE : KVQ_PLANE_K_SCALE;
  const int zp = which ? KVQ_PLANE_V_ZERO : KVQ_PLANE_K_ZERO;
  code_group32<BITS, SYM>(g, cp, sp, zp, b, h, t, g1, x1);
  code_group32<BITS, SYM>(g, cp, sp, zp, b, h, t, g2, x2);
}

template <int BN>
struct Smem {
  static constexpr int A_B = BM * BK * 2;            // 16 KB
  static constexpr int B_B = BN * BK * 2;            // up to 32 KB
  static constexpr int LA_B = 64 * BK * 2;           // LoRA A slice, up to 64 ranks (8 KB)
  static constexpr int STAGE_B = A_B + B_B + LA_B;
  static constexpr int U_OFF = kStages * STAGE_B;    // (alpha/r) x A^T as bf16 operand
  static constexpr int BP_OFF = U_OFF + BM * BK * 2; // B_p tile [BN][64 ranks]
  static constexpr int TOTAL = BP_OFF + BN * BK * 2 + 1024;   // + alignment slack
};

// NF4: W arrives as 4-bit NormalFloat codes; warps 4-11 (256 threads: one
// per tile row at BN = 256, two at BN = 128) turn each 64-input K slice into
// the bf16 tile the TMA would have landed (level x absmax in fp32, rounded
// once), 128-byte swizzled, and signal it on w_full; the x and A_p slices
// still come by TMA.
template <int BN, bool NF4>
__global__ void __launch_bounds__(NF4 ? kThreads + 32 * kDqWarps : kThreads, 1)
project_tc_kernel(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_w,
                  const __grid_constant__ CUtensorMap tm_a0, const __grid_constant__ CUtensorMap tm_a1,
                  const __grid_constant__ CUtensorMap tm_a2, const __grid_constant__ CUtensorMap tm_b0,
                  const __grid_constant__ CUtensorMap tm_b1, const __grid_constant__ CUtensorMap tm_b2,
                  const TcArgs args) {
  static_assert(!NF4 || BN == 128 || BN == 256, "256 dequantising threads cover the tile's rows");
  pdl_wait();
  pdl_trigger();
  using S = Smem<BN>;
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ uint64_t full_bar[kStages], empty_bar[kStages], w_full[kStages];
  __shared__ uint64_t u_bar, bp_bar, acc_bar;
  __shared__ float nf4_lv[16];
  __shared__ uint32_t tmem_base;
  __shared__ int fail;

  bool app_ok = true;                    // appending: the cache has room for the L tokens
  const int T0 = args.pack ? append_begin(args.g, args.L, &app_ok) : 0;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n0 = blockIdx.x * BN, m0 = blockIdx.y * BM;
  const int proj = n0 < args.n_off[1] ? 0 : n0 < args.n_off[2] ? 1 : 2;
  const int r = args.r[proj], rp = args.rp[proj];
  const CUtensorMap* tm_a = proj == 0 ? &tm_a0 : proj == 1 ? &tm_a1 : &tm_a2;
  const CUtensorMap* tm_b = proj == 0 ? &tm_b0 : proj == 1 ? &tm_b1 : &tm_b2;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&full_bar[i], 1);
      mbar_init(&empty_bar[i], 1);
      mbar_init(&w_full[i], kDqWarps);     // NF4: one arrival per dequantising warp
    }
    mbar_init(&u_bar, 1);
    mbar_init(&bp_bar, 1);
    mbar_init(&acc_bar, 1);
    fail = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (NF4 && threadIdx.x < 16) nf4_lv[threadIdx.x] = c_nf4_lv[threadIdx.x];
  if (warp == 1) {   // TMEM: 512 columns (main BN + LoRA <= 64)
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 512;"
                 ::"r"(smem_u32(&tmem_base)));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base;
  const uint32_t tmem_u = tmem + BN;
  const int KB = args.k_blocks;

  if (threadIdx.x == 0) {
    // ---------------- TMA producer ----------------
    if (r > 0) {
      mbar_expect_tx(&bp_bar, BN * BK * 2);
      tma_load_2d(smem + S::BP_OFF, tm_b, 0, n0 - args.n_off[proj], &bp_bar);
    }
    for (int kb = 0; kb < KB; ++kb) {
      const int s = kb % kStages;
      if (kb >= kStages && !mbar_wait(&empty_bar[s], ((kb / kStages) - 1) & 1)) {
        atomicOr(&fail, 1);
        break;
      }
      unsigned char* st = smem + s * S::STAGE_B;
      mbar_expect_tx(&full_bar[s], S::A_B + (NF4 ? 0 : S::B_B) + (r > 0 ? rp * BK * 2 : 0));
      tma_load_2d(st, &tm_x, kb * BK, m0, &full_bar[s]);
      if (!NF4)
        tma_load_2d(st + S::A_B, &tm_w, (args.kb_wrap ? kb % args.kb_wrap : kb) * BK, n0,
                    &full_bar[s]);
      if (r > 0) tma_load_2d(st + S::A_B + S::B_B, tm_a, kb * BK, 0, &full_bar[s]);
    }
  } else if (threadIdx.x == 32) {
    // ---------------- MMA issuer ----------------
    constexpr uint32_t id_main = idesc_bf16(BM, BN);
    const uint32_t id_u = idesc_bf16(BM, rp > 0 ? rp : 16);
    bool ok = true;
    for (int kb = 0; kb < KB; ++kb) {
      const int s = kb % kStages;
      if (!mbar_wait(&full_bar[s], (kb / kStages) & 1) ||
          (NF4 && !mbar_wait(&w_full[s], (kb / kStages) & 1))) {
        ok = false;
        break;
      }
      tc_fence_after();
      unsigned char* st = smem + s * S::STAGE_B;
#pragma unroll
      for (int kk = 0; kk < BK / 16; ++kk) {
        const uint64_t ad = sw128_desc(st + kk * 32);
        umma(tmem, ad, sw128_desc(st + S::A_B + kk * 32), id_main, (kb | kk) != 0);
        if (r > 0) umma(tmem_u, ad, sw128_desc(st + S::A_B + S::B_B + kk * 32), id_u, (kb | kk) != 0);
      }
      umma_commit(&empty_bar[s]);          // frees the stage when these MMAs finish
    }
    if (!ok) atomicOr(&fail, 1);
    umma_commit(&u_bar);                   // all main-loop MMAs done
  } else if (NF4 && warp >= 4) {
    // ---------- NF4 dequantisation: TPR threads per tile row ----------
    constexpr int TPR = 32 * kDqWarps / BN;               // 1 (BN = 256) or 2 (BN = 128)
    constexpr int NQ = 2 / TPR;                           // 16-byte code words per thread and slice
    const int dt = threadIdx.x - kThreads;                // 0 .. 255
    const int n = dt / TPR, h = dt % TPR;                 // row, part of the slice
    const int nkb = args.k_blocks;
    const uint8_t* crow = args.nf4_codes + (int64_t)(n0 + n) * (nkb * 32) + h * 16;
    const float* arow = args.nf4_absmax + (int64_t)(n0 + n) * nkb;
    // codes and absmax of this and the next two K slices in registers
    // (rotated each slice, so no array is indexed at run time)
    uint4 cq[3][NQ];
    float am[3];
#pragma unroll
    for (int i = 0; i < 3; ++i) {
#pragma unroll
      for (int q = 0; q < NQ; ++q) cq[i][q] = make_uint4(0, 0, 0, 0);
      am[i] = 0.f;
    }
    auto fetch = [&](int kb, uint4 (&x)[NQ], float& xa) {
      if (kb < KB) {
#pragma unroll
        for (int q = 0; q < NQ; ++q) x[q] = __ldg(reinterpret_cast<const uint4*>(crow + kb * 32 + 16 * q));
        xa = __ldg(arow + kb);
      }
    };
    fetch(0, cq[0], am[0]);
    fetch(1, cq[1], am[1]);
    const int rsw = (n >> 3) * 1024 + (n & 7) * 128;      // the row in the swizzled tile
    for (int kb = 0; kb < KB; ++kb) {
      const int s = kb % kStages;
      fetch(kb + 2, cq[2], am[2]);
      if (kb >= kStages) {                                // lane 0 waits for the slot, then the warp
        bool ok = true;
        if (lane == 0) ok = mbar_wait(&empty_bar[s], ((kb / kStages) - 1) & 1);
        if (!__shfl_sync(0xffffffffu, ok, 0)) {
          if (lane == 0) atomicOr(&fail, 1);
          break;
        }
      }
      unsigned char* wt = smem + s * S::STAGE_B + S::A_B;
      uint32_t w8[4 * NQ];
#pragma unroll
      for (int q = 0; q < NQ; ++q) {
        w8[4 * q] = cq[0][q].x; w8[4 * q + 1] = cq[0][q].y;
        w8[4 * q + 2] = cq[0][q].z; w8[4 * q + 3] = cq[0][q].w;
      }
      const float a = am[0];
#pragma unroll
      for (int q = 0; q < NQ; ++q) {
        cq[0][q] = cq[1][q];
        cq[1][q] = cq[2][q];
      }
      am[0] = am[1];
      am[1] = am[2];
      uint64_t a2;
      asm("mov.b64 %0, {%1, %1};" : "=l"(a2) : "f"(a));
#pragma unroll
      for (int j = 0; j < 4 * NQ; ++j) {                  // chunk c: inputs 8c .. 8c + 7
        const int c = 4 * NQ * h + j;
        uint32_t o[4];
        // byte offsets into the level table (4 x code) of the word's low and
        // high nibbles, four at a time
        const uint32_t lo4 = (w8[j] << 2) & 0x3C3C3C3Cu, hi4 = (w8[j] >> 2) & 0x3C3C3C3Cu;
#pragma unroll
        for (int i = 0; i < 4; ++i) {                     // byte i of word j: inputs 8c + 2i, + 1
          // the two levels times absmax as one packed fp32 multiply (each
          // product rounded as a scalar one would be), then one bf16 pair
          const char* lvb = reinterpret_cast<const char*>(nf4_lv);
          const uint32_t sel = 0x4440u | (uint32_t)i;     // byte i into byte 0, zeros above
          const float l0 = *reinterpret_cast<const float*>(lvb + __byte_perm(lo4, 0u, sel));
          const float l1 = *reinterpret_cast<const float*>(lvb + __byte_perm(hi4, 0u, sel));
          uint64_t p2, l2;
          asm("mov.b64 %0, {%1, %2};" : "=l"(l2) : "f"(l0), "f"(l1));
          asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(p2) : "l"(l2), "l"(a2));
          float q0, q1;
          asm("mov.b64 {%0, %1}, %2;" : "=f"(q0), "=f"(q1) : "l"(p2));
          o[i] = pack_bf16(q0, q1);
        }
        *reinterpret_cast<uint4*>(wt + rsw + ((c ^ (n & 7)) << 4)) = make_uint4(o[0], o[1], o[2], o[3]);
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");   // for the MMA's reads
      __syncwarp();
      if (lane == 0) mbar_arrive(&w_full[s]);
    }
  }
  // ---------------- (alpha/r) x A^T -> bf16 operand in shared memory ----------
  const bool u_ok = __syncthreads_and(mbar_wait(&u_bar, 0)) != 0;   // uniform
  tc_fence_after();
  const int row = warp * 32 + lane;            // TMEM lane = tile row
  const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
  if (r > 0 && u_ok && warp < 4) {
    unsigned char* us = smem + S::U_OFF;
    for (int c0 = 0; c0 < rp; c0 += 16) {
      float v[16];
      tmem_ld16(tmem_u + lane_base + c0, v);
      uint32_t w[8];
#pragma unroll
      for (int i = 0; i < 8; ++i)
        w[i] = pack_bf16(v[2 * i] * args.alpha_over_r, v[2 * i + 1] * args.alpha_over_r);
      // two 16-byte chunks (k = c0 .. c0+7, c0+8 .. c0+15) of row `row`,
      // placed at chunk index c ^ (row % 8) of the 128-byte row
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int chunk = (c0 / 8 + h) ^ (row & 7);
        *reinterpret_cast<uint4*>(us + row * 128 + chunk * 16) =
            make_uint4(w[4 * h], w[4 * h + 1], w[4 * h + 2], w[4 * h + 3]);
      }
    }
    // ranks rp .. 63 of the operand row are never read (the MMA uses K = rp)
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  tc_fence_before();
  __syncthreads();
  if (!u_ok && threadIdx.x == 0) atomicOr(&fail, 1);
  if (threadIdx.x == 32) {
    tc_fence_after();
    if (r > 0 && u_ok && !fail) {
      if (mbar_wait(&bp_bar, 0)) {
        const uint32_t id_main = idesc_bf16(BM, BN);
        for (int kk = 0; kk < rp / 16; ++kk)
          umma(tmem, sw128_desc(smem + S::U_OFF + kk * 32),
               sw128_desc(smem + S::BP_OFF + kk * 32), id_main, 1);
      } else {
        atomicOr(&fail, 1);
      }
    }
    umma_commit(&acc_bar);
  }
  // ---------------- epilogue: RoPE and head-major store ----------------
  const bool acc_wait = mbar_wait(&acc_bar, 0);
  const bool good = __syncthreads_and(acc_wait) && !*reinterpret_cast<volatile int*>(&fail);
  tc_fence_after();
  const int m = m0 + row;
  const bool active = m < args.M;                     // rows past M: load, do not store
  if (good && warp < 4) {
    const int D = args.D, half = D / 2;
    const int mm = active ? m : 0;
    const int b = mm / args.L, l = mm % args.L;
    const int H = proj == 0 ? args.Hq : args.Hkv;
    const int col0 = n0 - args.n_off[proj];           // first column within projection
    __nv_bfloat16* out = reinterpret_cast<__nv_bfloat16*>(args.out[proj]);
    const bool rope = args.rope && proj < 2;
    const int pos = args.pos0 + pos_of(args.pos_dev, args.pos_stride, b) + l;
    if (args.plain_out) {
      // plain product: the accumulator row as fp32
      const int N = args.n_off[3];
      for (int c = 0; c < BN; c += 16) {
        float v[16];
        tmem_ld16(tmem + lane_base + c, v);
        if (!active) continue;
        float4* d = reinterpret_cast<float4*>(args.plain_out + (int64_t)m * N + n0 + c);
#pragma unroll
        for (int i = 0; i < 4; ++i) d[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
      }
    } else if (args.pack && proj > 0) {
      // append: k (after RoPE) and v rounded to bf16, then coded per token
      // in groups of 32 channels straight into the cache planes
      const Geom& gg = args.g;
      const int bits = proj == 1 ? gg.kb : gg.vb;
      const bool sym = gg.fmt == KVQ_FMT_SYMMETRIC;
      const int t = T0 + l;
      for (int hc = 0; hc < BN; hc += D) {
        const int head = (col0 + hc) / D;
        for (int j = 0; j < half; j += 32) {
          float x1[32], x2[32];
#pragma unroll
          for (int u = 0; u < 32; u += 16) {
            tmem_ld16(tmem + lane_base + hc + j + u, x1 + u);
            tmem_ld16(tmem + lane_base + hc + half + j + u, x2 + u);
            if (rope) {
#pragma unroll
              for (int i = 0; i < 16; ++i) {
                float c, sn;
                rope_cs(pos, args.theta_hi[j + u + i], args.theta_lo[j + u + i], &c, &sn);
                rope_rot(x1[u + i], x2[u + i], c, sn);
              }
            }
          }
          if (!active || !app_ok) continue;
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            x1[i] = __bfloat162float(__float2bfloat16_rn(x1[i]));
            x2[i] = __bfloat162float(__float2bfloat16_rn(x2[i]));
          }
          const int g1 = j / 32, g2 = (half + j) / 32, which = proj - 1;
          if (sym) {
            if (bits == 2) code_pair<2, true>(gg, which, b, head, t, g1, g2, x1, x2);
            else if (bits == 4) code_pair<4, true>(gg, which, b, head, t, g1, g2, x1, x2);
            else code_pair<8, true>(gg, which, b, head, t, g1, g2, x1, x2);
          } else {
            if (bits == 2) code_pair<2, false>(gg, which, b, head, t, g1, g2, x1, x2);
            else if (bits == 4) code_pair<4, false>(gg, which, b, head, t, g1, g2, x1, x2);
            else code_pair<8, false>(gg, which, b, head, t, g1, g2, x1, x2);
          }
        }
      }
    } else
    for (int j = 0; j < half; j += 16) {              // 16 frequencies at a time
      float cs[16], sn[16];
      if (rope) {
#pragma unroll
        for (int i = 0; i < 16; ++i)
          rope_cs(pos, args.theta_hi[j + i], args.theta_lo[j + i], &cs[i], &sn[i]);
      }
      for (int hc = 0; hc < BN; hc += D) {            // whole heads in the tile
        const int head = (col0 + hc) / D;
        __nv_bfloat16* orow = out + (((int64_t)b * H + head) * args.L + l) * D;
        float x1[16], x2[16];
        tmem_ld16(tmem + lane_base + hc + j, x1);
        tmem_ld16(tmem + lane_base + hc + half + j, x2);
        if (rope) {
#pragma unroll
          for (int i = 0; i < 16; ++i) rope_rot(x1[i], x2[i], cs[i], sn[i]);
        }
        if (!active) continue;
        uint32_t w1[8], w2[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          w1[i] = pack_bf16(x1[2 * i], x1[2 * i + 1]);
          w2[i] = pack_bf16(x2[2 * i], x2[2 * i + 1]);
        }
        uint4* d1 = reinterpret_cast<uint4*>(orow + j);
        uint4* d2 = reinterpret_cast<uint4*>(orow + half + j);
        d1[0] = make_uint4(w1[0], w1[1], w1[2], w1[3]);
        d1[1] = make_uint4(w1[4], w1[5], w1[6], w1[7]);
        d2[0] = make_uint4(w2[0], w2[1], w2[2], w2[3]);
        d2[1] = make_uint4(w2[4], w2[5], w2[6], w2[7]);
      }
    }
  }
  if (threadIdx.x == 0 && !good) atomicOr(args.err, 2);
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 512;" ::"r"(tmem));
  }
  // appending: the last CTA to arrive advances the cache's token count
  if (args.pack) quant::append_arrive_spread(args.g.state, T0, args.L, app_ok);
}

// ---------------------------------------------------------------------------
// host: tensor maps through the driver entry point (no libcuda link)
// ---------------------------------------------------------------------------
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// 2D bf16 tensor [rows][cols] (cols contiguous), box [box_rows][64 cols],
// 128-byte swizzle; out-of-range elements read as zero.
bool make_map(CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult res = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                    box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return res == CUDA_SUCCESS;
}

template <int BN, bool NF4 = false>
cudaError_t launch_bn(const CUtensorMap maps[8], const TcArgs& a, cudaStream_t s) {
  const int smem = Smem<BN>::TOTAL;
  auto kern = project_tc_kernel<BN, NF4>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  dim3 grid(a.n_off[3] / BN, (a.M + BM - 1) / BM);
  launch_pdl(kern, dim3(grid), dim3(NF4 ? kThreads + 32 * kDqWarps : kThreads), smem, s, maps[0], maps[1], maps[2], maps[3], maps[4], maps[5],
                                    maps[6], maps[7], a);
  return cudaGetLastError();
}

}  // namespace

// Tile width for these head counts, or 0 if the tensor-core path does not
// cover the shape (then the caller uses the SIMT kernel).
int project_tc_tile(int Hq, int Hkv, int D, int d_in) {
  if (d_in % 64) return 0;
  const int nq = Hq * D, nk = Hkv * D;
  for (int bn : {256, 128}) {
    if (bn < D) continue;
    if (nq % bn == 0 && nk % bn == 0) return bn;
  }
  return 0;
}

// NF4 base (codes, absmax) when `w` is null.
static cudaError_t launch_tc(const void* x, int B, int L, int d_in, const void* w,
                             const uint8_t* nf4_codes, const float* nf4_absmax,
                             const void* const a[3], const void* const bm[3], const int r[3],
                             float alpha_over_r, int Hq, int Hkv, int D, int pos0,
                             const int* pos_dev, float rope_base, void* const out[3], int* err,
                             cudaStream_t s, const Geom* append_to, int pos_stride) {
  const bool nf4 = w == nullptr;
  const int bn = project_tc_tile(Hq, Hkv, D, d_in);
  if (!bn) return cudaErrorNotSupported;
  TcArgs t;
  t.nf4_codes = nf4_codes;
  t.nf4_absmax = nf4_absmax;
  t.plain_out = nullptr;
  t.kb_wrap = 0;
  t.pack = append_to != nullptr;
  if (append_to) t.g = *append_to;
  else memset(&t.g, 0, sizeof t.g);
  const int M = B * L;
  for (int i = 0; i < 3; ++i) {
    t.out[i] = out[i];
    t.r[i] = r[i];
    t.rp[i] = (r[i] + 15) / 16 * 16;
  }
  t.B = B; t.L = L; t.M = M; t.D = D; t.Hq = Hq; t.Hkv = Hkv;
  t.n_off[0] = 0; t.n_off[1] = Hq * D; t.n_off[2] = (Hq + Hkv) * D; t.n_off[3] = (Hq + 2 * Hkv) * D;
  t.pos0 = pos0; t.pos_dev = pos_dev; t.pos_stride = pos_stride; t.alpha_over_r = alpha_over_r;
  t.rope = rope_base > 0.f; t.k_blocks = d_in / 64; t.err = err;
  rope_theta_table(rope_base, D, t.theta_hi, t.theta_lo);
  CUtensorMap maps[8];
  bool ok = make_map(&maps[0], x, M, d_in, BM);
  if (nf4) maps[1] = maps[0];                       // unused: any valid map
  else ok = ok && make_map(&maps[1], w, (uint64_t)t.n_off[3], d_in, bn);
  const int dout[3] = {Hq * D, Hkv * D, Hkv * D};
  for (int p = 0; p < 3 && ok; ++p) {
    if (r[p] > 0) {
      ok = make_map(&maps[2 + p], a[p], r[p], d_in, t.rp[p]) &&
           make_map(&maps[5 + p], bm[p], dout[p], r[p], bn);
    } else {  // unused: any valid map
      maps[2 + p] = maps[0];
      maps[5 + p] = maps[0];
    }
  }
  if (!ok) return cudaErrorInvalidValue;
  if (nf4) return bn == 256 ? launch_bn<256, true>(maps, t, s) : launch_bn<128, true>(maps, t, s);
  return bn == 256 ? launch_bn<256>(maps, t, s) : launch_bn<128>(maps, t, s);
}

cudaError_t launch_project_tc(const void* x, int B, int L, int d_in, const void* w,
                              const void* const a[3], const void* const bm[3], const int r[3],
                              float alpha_over_r, int Hq, int Hkv, int D, int pos0,
                              const int* pos_dev, float rope_base, void* const out[3], int* err,
                              cudaStream_t s, const Geom* append_to, int pos_stride) {
  if (!w) return cudaErrorInvalidValue;
  return launch_tc(x, B, L, d_in, w, nullptr, nullptr, a, bm, r, alpha_over_r, Hq, Hkv, D, pos0,
                   pos_dev, rope_base, out, err, s, append_to, pos_stride);
}

// C [M][N] fp32 = A [M][K] B^T on tcgen05, A bf16 K-major, B's rows bf16 of Kb
// elements repeated along K (K a multiple of Kb: B(k) = Bt[:, k mod Kb]).
cudaError_t launch_gemm_tc_bf16(const void* a, int M, int K, const void* bt, int N, int Kb,
                                float* c, int* err, cudaStream_t s) {
  if (M <= 0 || N <= 0 || K <= 0 || K % 64 || Kb % 64 || K % Kb) return cudaErrorInvalidValue;
  const int bn = N % 256 == 0 ? 256 : N % 128 == 0 ? 128 : 0;
  if (!bn) return cudaErrorNotSupported;
  TcArgs t;
  memset(&t, 0, sizeof t);
  t.B = 1; t.L = M; t.M = M; t.D = 64; t.Hq = N / 64; t.Hkv = 1;
  t.n_off[0] = 0; t.n_off[1] = N; t.n_off[2] = N; t.n_off[3] = N;
  t.k_blocks = K / 64; t.kb_wrap = Kb / 64 == K / 64 ? 0 : Kb / 64; t.err = err;
  t.plain_out = c;
  CUtensorMap maps[8];
  if (!make_map(&maps[0], a, M, K, BM) || !make_map(&maps[1], bt, N, Kb, bn))
    return cudaErrorInvalidValue;
  for (int i = 2; i < 8; ++i) maps[i] = maps[0];   // unused: no adapters
  return bn == 256 ? launch_bn<256>(maps, t, s) : launch_bn<128>(maps, t, s);
}

bool project_tc_nf4_supported(int Hq, int Hkv, int D, int d_in) {
  return project_tc_tile(Hq, Hkv, D, d_in) != 0;
}

cudaError_t launch_project_tc_nf4(const void* x, int B, int L, int d_in, const void* codes,
                                  const void* absmax, const void* const a[3],
                                  const void* const bm[3], const int r[3], float alpha_over_r,
                                  int Hq, int Hkv, int D, int pos0, const int* pos_dev,
                                  float rope_base, void* const out[3], int* err, cudaStream_t s,
                                  int pos_stride) {
  return launch_tc(x, B, L, d_in, nullptr, static_cast<const uint8_t*>(codes),
                   static_cast<const float*>(absmax), a, bm, r, alpha_over_r, Hq, Hkv, D, pos0,
                   pos_dev, rope_base, out, err, s, nullptr, pos_stride);
}

}  // namespace kvq
