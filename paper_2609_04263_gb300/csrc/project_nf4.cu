// LoRA-adapted Q/K/V projection over a frozen NF4 base (Sections 3.4 and 4:
// the reported Gemma and Llama-3.1 runs keep NF4 bases and explicit rank-r
// branches; Section 2 cites QLoRA's 4-bit NormalFloat for such bases):
//   y = x dequant(W)^T + (alpha/r) (x A_p^T) B_p^T,   then RoPE on q and k,
// where a base weight is level[code] * absmax, one 4-bit code per weight and
// one fp32 absmax per block of 64 consecutive inputs of a row.
//
// The base is dequantized in the GEMM's operand path: per 64-input K tile the
// CTA copies its 128 rows' codes (32 bytes each) and absmax values with
// cp.async, turns them into a bf16 tile in shared memory (level from a
// shared-memory table, times absmax, rounded to bf16) and feeds it to
// mma.sync m16n8k16 as the B operand; x and the LoRA A_p rows come through the
// same 3-stage ring.  x A_p^T accumulates beside the main product, is scaled
// by alpha/r and rounded to bf16, and one more pass adds (alpha/r)(x A_p^T) B_p^T.
// The epilogue stages the fp32 tile in shared memory, applies rotate-half
// RoPE and stores head-major bf16.  BM = 64 rows per CTA for prefill, 16 for
// decode rows; 128 output features per CTA, inside one projection.
#include <math.h>

#include "decode_attn.cuh"
#include "proj_decode.cuh"

namespace kvq {
namespace {

constexpr int NBN = 128;             // output features per CTA
constexpr int NBK = 64;              // inputs per K tile (one NF4 block)
constexpr int kNStages = 3;
constexpr int kNThreads = 256;       // 8 warps
constexpr int LDP = 72;              // padded shared-memory row (bf16 elements)

// The 16 NF4 levels, code 0 .. 15, as QLoRA publishes the data type.
__constant__ float c_nf4_levels[16] = {
    -1.0f, -0.6961928009986877f, -0.5250730514526367f, -0.39491748809814453f,
    -0.28444138169288635f, -0.18477343022823334f, -0.09105003625154495f, 0.0f,
    0.07958029955625534f, 0.16093020141124725f, 0.24611230194568634f, 0.33791524171829224f,
    0.44070982933044434f, 0.5626170039176941f, 0.7229568362236023f, 1.0f};

struct Nf4Args {
  const __nv_bfloat16* x;
  const uint8_t* codes;        // [N][d_in / 2]
  const float* absmax;         // [N][d_in / 64]
  const __nv_bfloat16* a[3];   // [r_p][d_in]
  const __nv_bfloat16* bm[3];  // [d_out_p][r_p]
  int r[3];
  __nv_bfloat16* out[3];
  int B, L, M, d_in, Hq, Hkv, D;
  int n_off[4];
  int pos0;
  const int* pos_dev;
  int pos_stride;
  float alpha_over_r;
  int rope;
  float theta_hi[128], theta_lo[128];
};

template <int BM>
struct Nf4Cfg {
  static constexpr int WM = BM == 64 ? 2 : 1;             // warps along rows
  static constexpr int WN = 8 / WM;                       // warps along features
  static constexpr int MT = BM / (16 * WM);               // m16 tiles per warp
  static constexpr int NT = NBN / (8 * WN);               // n8 tiles per warp
  static constexpr int X_B = BM * LDP * 2;
  static constexpr int A_B = 64 * LDP * 2;                // up to 64 LoRA ranks
  static constexpr int C_B = NBN * NBK / 2;               // codes
  static constexpr int S_B = NBN * 4;                     // absmax
  static constexpr int STAGE = X_B + A_B + C_B + S_B;
  static constexpr int WD_OFF = kNStages * STAGE;         // dequantized W tile [128][LDP]
  static constexpr int U_OFF = WD_OFF + NBN * LDP * 2;    // (alpha/r) x A^T as bf16 [BM][LDP]
  static constexpr int BP_OFF = U_OFF + BM * LDP * 2;     // B_p rows [128][LDP]
  static constexpr int TOTAL = BP_OFF + NBN * LDP * 2;
  static constexpr int CT_LD = NBN + 4;                   // epilogue fp32 tile, over the stages
  static_assert(BM * CT_LD * 4 <= kNStages * STAGE, "epilogue tile fits the ring");
};

__device__ __forceinline__ void cp_async16(void* dst, const void* src, bool valid) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;"
               ::"r"(dattn::smem_u32(dst)), "l"(src), "r"(valid ? 16 : 0) : "memory");
}
__device__ __forceinline__ void cp_async4(void* dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;"
               ::"r"(dattn::smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

__device__ __forceinline__ void ldsm_x4(const void* p, uint32_t r[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]) : "r"(dattn::smem_u32(p)));
}
__device__ __forceinline__ void ldsm_x2(const void* p, uint32_t r[2]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0,%1}, [%2];"
               : "=r"(r[0]), "=r"(r[1]) : "r"(dattn::smem_u32(p)));
}

template <int BM>
__global__ void __launch_bounds__(kNThreads)
project_nf4_kernel(const Nf4Args args) {
  pdl_wait();
  pdl_trigger();
  using C = Nf4Cfg<BM>;
  extern __shared__ __align__(128) unsigned char smem[];
  __shared__ float lv[16];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int gid = lane >> 2, tq = lane & 3;
  const int wm = warp / C::WN, wn = warp % C::WN;
  const int n0 = blockIdx.x * NBN, m0 = blockIdx.y * BM;
  const int proj = n0 < args.n_off[1] ? 0 : n0 < args.n_off[2] ? 1 : 2;
  const int r = args.r[proj];
  const __nv_bfloat16* ap = args.a[proj];
  const int d_in = args.d_in, nkt = d_in / NBK;
  if (tid < 16) lv[tid] = c_nf4_levels[tid];

  // ---- one K tile's copies into stage s ----
  auto load_stage = [&](int kt, int s) {
    unsigned char* st = smem + s * C::STAGE;
    const int k0 = kt * NBK;
    for (int i = tid; i < BM * 8; i += kNThreads) {               // x: BM rows x 8 chunks
      const int row = i >> 3, ch = i & 7, m = m0 + row;
      const bool ok = m < args.M;
      cp_async16(st + row * LDP * 2 + ch * 16, args.x + (int64_t)(ok ? m : 0) * d_in + k0 + ch * 8, ok);
    }
    for (int i = tid; i < r * 8; i += kNThreads) {                 // A_p: r rows x 8 chunks
      const int row = i >> 3, ch = i & 7;
      cp_async16(st + C::X_B + row * LDP * 2 + ch * 16, ap + (int64_t)row * d_in + k0 + ch * 8, true);
    }
    {                                                              // codes: 128 rows x 2 chunks
      const int row = tid >> 1, ch = tid & 1;
      cp_async16(st + C::X_B + C::A_B + row * 32 + ch * 16,
                 args.codes + (int64_t)(n0 + row) * (d_in / 2) + kt * 32 + ch * 16, true);
    }
    if (tid < NBN)                                                 // absmax of the block
      cp_async4(st + C::X_B + C::A_B + C::C_B + tid * 4,
                args.absmax + (int64_t)(n0 + tid) * nkt + kt);
  };

  float acc[C::MT][C::NT][4];
  float uacc[C::MT][2][4];
#pragma unroll
  for (int i = 0; i < C::MT; ++i) {
#pragma unroll
    for (int j = 0; j < C::NT; ++j) acc[i][j][0] = acc[i][j][1] = acc[i][j][2] = acc[i][j][3] = 0.f;
#pragma unroll
    for (int j = 0; j < 2; ++j) uacc[i][j][0] = uacc[i][j][1] = uacc[i][j][2] = uacc[i][j][3] = 0.f;
  }
  const int ut = r / 8;                                           // rank n8 tiles
  unsigned char* wd = smem + C::WD_OFF;

#pragma unroll
  for (int s = 0; s < kNStages - 1; ++s) {
    if (s < nkt) load_stage(s, s);
    cp_commit();
  }
  for (int kt = 0; kt < nkt; ++kt) {
    cp_wait<kNStages - 2>();
    __syncthreads();                                   // stage kt landed; W tile kt - 1 consumed
    const unsigned char* st = smem + (kt % kNStages) * C::STAGE;
    // dequantize the tile's base weights: thread = (row, half of the 64 inputs)
    {
      const int row = tid >> 1, half = tid & 1;
      const uint4 cw = *reinterpret_cast<const uint4*>(st + C::X_B + C::A_B + row * 32 + half * 16);
      const float am = *reinterpret_cast<const float*>(st + C::X_B + C::A_B + C::C_B + row * 4);
      const uint32_t w4[4] = {cw.x, cw.y, cw.z, cw.w};
      uint32_t o[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) {                   // byte i: inputs 2i (low nibble), 2i + 1
        const uint32_t byte = (w4[i >> 2] >> (8 * (i & 3))) & 0xFFu;
        o[i] = dattn::pack_bf16(lv[byte & 15u] * am, lv[byte >> 4] * am);
      }
      uint4* dst = reinterpret_cast<uint4*>(wd + row * LDP * 2 + half * 64);
#pragma unroll
      for (int i = 0; i < 4; ++i) dst[i] = make_uint4(o[4 * i], o[4 * i + 1], o[4 * i + 2], o[4 * i + 3]);
    }
    // next tile's copies (into the stage consumed two tiles ago)
    if (kt + kNStages - 1 < nkt) load_stage(kt + kNStages - 1, (kt + kNStages - 1) % kNStages);
    cp_commit();
    __syncthreads();                                   // W tile kt ready
    const unsigned char* xs = st;
    const unsigned char* as = st + C::X_B;
#pragma unroll
    for (int kk = 0; kk < NBK / 16; ++kk) {
      uint32_t af[C::MT][4];
#pragma unroll
      for (int mt = 0; mt < C::MT; ++mt) {
        const int row = wm * (16 * C::MT) + mt * 16 + (lane & 15);
        ldsm_x4(xs + row * LDP * 2 + (kk * 16 + (lane >> 4) * 8) * 2, af[mt]);
      }
#pragma unroll
      for (int nt = 0; nt < C::NT; ++nt) {
        uint32_t bf[2];
        const int nrow = wn * (8 * C::NT) + nt * 8 + (lane & 7);
        ldsm_x2(wd + nrow * LDP * 2 + (kk * 16 + ((lane >> 3) & 1) * 8) * 2, bf);
#pragma unroll
        for (int mt = 0; mt < C::MT; ++mt) dattn::mma16816(acc[mt][nt], af[mt], bf[0], bf[1]);
      }
      // x A_p^T: rank tiles wn, wn + WN (at most 2 per warp)
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const int t8 = wn + u * C::WN;
        if (t8 >= ut) continue;
        uint32_t bf[2];
        const int nrow = t8 * 8 + (lane & 7);
        ldsm_x2(as + nrow * LDP * 2 + (kk * 16 + ((lane >> 3) & 1) * 8) * 2, bf);
#pragma unroll
        for (int mt = 0; mt < C::MT; ++mt) dattn::mma16816(uacc[mt][u], af[mt], bf[0], bf[1]);
      }
    }
  }
  cp_wait<0>();
  __syncthreads();

  // ---- rank-r branch: U = (alpha/r) x A_p^T as bf16, then y += U B_p^T ----
  const int rp = (r + 15) / 16 * 16;
  if (r > 0) {
    unsigned char* us = smem + C::U_OFF;
    unsigned char* bp = smem + C::BP_OFF;
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      const int t8 = wn + u * C::WN;
      if (t8 >= ut) continue;
#pragma unroll
      for (int mt = 0; mt < C::MT; ++mt)
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int row = wm * (16 * C::MT) + mt * 16 + gid + 8 * h;
          *reinterpret_cast<uint32_t*>(us + row * LDP * 2 + (t8 * 8 + 2 * tq) * 2) =
              dattn::pack_bf16(uacc[mt][u][2 * h] * args.alpha_over_r,
                               uacc[mt][u][2 * h + 1] * args.alpha_over_r);
        }
    }
    if (r < rp) {                                       // zero the pad ranks of U and B_p
      for (int i = tid; i < BM; i += kNThreads)
        *reinterpret_cast<uint4*>(us + i * LDP * 2 + r * 2) = make_uint4(0, 0, 0, 0);
      for (int i = tid; i < NBN; i += kNThreads)
        *reinterpret_cast<uint4*>(bp + i * LDP * 2 + r * 2) = make_uint4(0, 0, 0, 0);
    }
    const __nv_bfloat16* bm = args.bm[proj] + (int64_t)(n0 - args.n_off[proj]) * r;
    for (int i = tid; i < NBN * (r / 8); i += kNThreads) {
      const int row = i / (r / 8), ch = i % (r / 8);
      cp_async16(bp + row * LDP * 2 + ch * 16, bm + (int64_t)row * r + ch * 8, true);
    }
    cp_commit();
    cp_wait<0>();
    __syncthreads();
    for (int kk = 0; kk < rp / 16; ++kk) {
      uint32_t af[C::MT][4];
#pragma unroll
      for (int mt = 0; mt < C::MT; ++mt) {
        const int row = wm * (16 * C::MT) + mt * 16 + (lane & 15);
        ldsm_x4(us + row * LDP * 2 + (kk * 16 + (lane >> 4) * 8) * 2, af[mt]);
      }
#pragma unroll
      for (int nt = 0; nt < C::NT; ++nt) {
        uint32_t bf[2];
        const int nrow = wn * (8 * C::NT) + nt * 8 + (lane & 7);
        ldsm_x2(bp + nrow * LDP * 2 + (kk * 16 + ((lane >> 3) & 1) * 8) * 2, bf);
#pragma unroll
        for (int mt = 0; mt < C::MT; ++mt) dattn::mma16816(acc[mt][nt], af[mt], bf[0], bf[1]);
      }
    }
    __syncthreads();
  }

  // ---- epilogue: fp32 tile through shared memory, RoPE, head-major bf16 ----
  float* ct = reinterpret_cast<float*>(smem);
#pragma unroll
  for (int mt = 0; mt < C::MT; ++mt)
#pragma unroll
    for (int nt = 0; nt < C::NT; ++nt)
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int row = wm * (16 * C::MT) + mt * 16 + gid + 8 * h;
        const int col = wn * (8 * C::NT) + nt * 8 + 2 * tq;
        *reinterpret_cast<float2*>(ct + row * C::CT_LD + col) =
            make_float2(acc[mt][nt][2 * h], acc[mt][nt][2 * h + 1]);
      }
  __syncthreads();
  const int D = args.D, half = D / 2;
  const int H = proj == 0 ? args.Hq : args.Hkv;
  const int col0 = n0 - args.n_off[proj];
  const bool rope = args.rope && proj < 2;
  // work items: (row, head of the tile, 8 frequencies)
  const int per_row = (NBN / D) * (half / 8);
  for (int it = tid; it < BM * per_row; it += kNThreads) {
    const int row = it / per_row, rem = it % per_row;
    const int hd = rem / (half / 8), f0 = (rem % (half / 8)) * 8;
    const int m = m0 + row;
    if (m >= args.M) continue;
    const int b = m / args.L, l = m % args.L;
    const float* c1 = ct + row * C::CT_LD + hd * D + f0;
    float x1[8], x2[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      x1[i] = c1[i];
      x2[i] = c1[half + i];
    }
    if (rope) {
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        float cs, sn;
        pdec::rope_cos_sin(args.pos0 + pos_of(args.pos_dev, args.pos_stride, b) + l,
                           args.theta_hi[f0 + i], args.theta_lo[f0 + i], &cs, &sn);
        const float a = x1[i], bb = x2[i];
        x1[i] = a * cs - bb * sn;
        x2[i] = bb * cs + a * sn;
      }
    }
    const int head = (col0 + hd * D) / D;
    __nv_bfloat16* orow = args.out[proj] + (((int64_t)b * H + head) * args.L + l) * D;
    uint32_t w1[4], w2[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      w1[i] = dattn::pack_bf16(x1[2 * i], x1[2 * i + 1]);
      w2[i] = dattn::pack_bf16(x2[2 * i], x2[2 * i + 1]);
    }
    *reinterpret_cast<uint4*>(orow + f0) = make_uint4(w1[0], w1[1], w1[2], w1[3]);
    *reinterpret_cast<uint4*>(orow + half + f0) = make_uint4(w2[0], w2[1], w2[2], w2[3]);
  }
}

template <int BM>
cudaError_t launch_nf4_bm(const Nf4Args& a, cudaStream_t s) {
  auto kern = project_nf4_kernel<BM>;
  const int smem = Nf4Cfg<BM>::TOTAL;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  dim3 grid(a.n_off[3] / NBN, (a.M + BM - 1) / BM);
  launch_pdl(kern, grid, dim3(kNThreads), (size_t)smem, s, a);
  return cudaGetLastError();
}

}  // namespace

bool project_nf4_supported(int d_in, int Hq, int Hkv, int D, const int r[3]) {
  if (d_in <= 0 || d_in % NBK) return false;
  if (D != 64 && D != 128) return false;
  if ((Hq * D) % NBN || (Hkv * D) % NBN) return false;
  for (int p = 0; p < 3; ++p)
    if (r[p] < 0 || r[p] > 64 || r[p] % 8) return false;
  return true;
}

cudaError_t launch_project_nf4(const void* x, int B, int L, int d_in, const void* codes,
                               const void* absmax, const void* const a[3],
                               const void* const bm[3], const int r[3], float alpha_over_r,
                               int Hq, int Hkv, int D, int pos0, const int* pos_dev,
                               float rope_base, void* const out[3], cudaStream_t s,
                               int pos_stride) {
  Nf4Args t;
  t.x = static_cast<const __nv_bfloat16*>(x);
  t.codes = static_cast<const uint8_t*>(codes);
  t.absmax = static_cast<const float*>(absmax);
  for (int p = 0; p < 3; ++p) {
    t.a[p] = static_cast<const __nv_bfloat16*>(a[p]);
    t.bm[p] = static_cast<const __nv_bfloat16*>(bm[p]);
    t.r[p] = r[p];
    t.out[p] = static_cast<__nv_bfloat16*>(out[p]);
  }
  t.B = B; t.L = L; t.M = B * L; t.d_in = d_in; t.Hq = Hq; t.Hkv = Hkv; t.D = D;
  t.n_off[0] = 0; t.n_off[1] = Hq * D; t.n_off[2] = (Hq + Hkv) * D; t.n_off[3] = (Hq + 2 * Hkv) * D;
  t.pos0 = pos0; t.pos_dev = pos_dev; t.pos_stride = pos_stride; t.alpha_over_r = alpha_over_r;
  t.rope = rope_base > 0.f;
  rope_theta_table(rope_base, D, t.theta_hi, t.theta_lo);
  return t.M <= 16 ? launch_nf4_bm<16>(t, s) : launch_nf4_bm<64>(t, s);
}

}  // namespace kvq
