// LoRA-adapted Q/K/V projection (Section 3, Eq. 1 and Eq. lora) with rotary
// positions, written head-major.  The adapter stays an explicit rank-r
// branch (Section 3.4): y = x W^T + (alpha/r) (x A^T) B^T.
#include <math.h>

#include "proj_decode.cuh"

namespace kvq {
// The weight-streaming decode projection (proj_stream.cu); cudaErrorNotSupported
// when the shape is outside its range (M > 16, d_in > 4096, rank > 64).
cudaError_t launch_project_decode_stream(const pdec::ProjArgs& p, int* err, cudaStream_t s);
}  // namespace kvq

namespace kvq {
namespace {
using namespace pdec;

constexpr int kMT = 32;     // rows per CTA
constexpr int kKC = 32;     // k chunk
constexpr int kThreads = 256;

// One CTA: kMT rows of x times one head's D output columns.
__global__ void __launch_bounds__(kThreads) project_simt_kernel(ProjArgs p) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ float sm[];
  const int D = p.D, M = p.B * p.L;
  const int hh = blockIdx.y;                 // stacked head index over q, k, v
  const int proj = hh < p.Hq ? 0 : hh < p.Hq + p.Hkv ? 1 : 2;
  const int head = proj == 0 ? hh : proj == 1 ? hh - p.Hq : hh - p.Hq - p.Hkv;
  const int r = p.r[proj];
  const int m0 = blockIdx.x * kMT;
  float* Xs = sm;                            // [kMT][kKC+1]
  float* Ws = Xs + kMT * (kKC + 1);          // [max(D, 64)][kKC+1]
  float* U = Ws + 256 * (kKC + 1);           // [kMT][64]
  float* Y = U + kMT * 64;                   // [kMT][D]
  const int rg = kThreads / D > 0 ? kThreads / D : 1;   // row groups
  const int col = threadIdx.x % D, rgi = threadIdx.x / D;
  const int rows_per = kMT / rg;
  float acc[32];
#pragma unroll
  for (int i = 0; i < 32; ++i) acc[i] = 0.f;
  float uacc[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) uacc[i] = 0.f;

  // x A^T (rank-r down projection), (m, j) pairs spread over the threads
  if (r > 0) {
    for (int k0 = 0; k0 < p.d_in; k0 += kKC) {
      for (int i = threadIdx.x; i < kMT * kKC; i += kThreads) {
        const int m = i / kKC, k = i % kKC;
        const int gm = m0 + m;
        Xs[m * (kKC + 1) + k] = (gm < M && k0 + k < p.d_in)
            ? ld_act(p.x, (int64_t)gm * p.d_in + k0 + k, p.act) : 0.f;
      }
      for (int i = threadIdx.x; i < r * kKC; i += kThreads) {
        const int j = i / kKC, k = i % kKC;
        Ws[j * (kKC + 1) + k] = k0 + k < p.d_in
            ? ld_act(p.a[proj], (int64_t)j * p.d_in + k0 + k, p.act) : 0.f;
      }
      __syncthreads();
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int idx = threadIdx.x + u * kThreads;
        if (idx < kMT * r) {
          const int m = idx / r, j = idx % r;
          float a = uacc[u];
          for (int k = 0; k < kKC; ++k) a += Xs[m * (kKC + 1) + k] * Ws[j * (kKC + 1) + k];
          uacc[u] = a;
        }
      }
      __syncthreads();
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int idx = threadIdx.x + u * kThreads;
      if (idx < kMT * r) U[(idx / r) * 64 + idx % r] = uacc[u] * p.alpha_over_r;
    }
  }
  // x W^T for this head's rows of W
  for (int k0 = 0; k0 < p.d_in; k0 += kKC) {
    for (int i = threadIdx.x; i < kMT * kKC; i += kThreads) {
      const int m = i / kKC, k = i % kKC;
      const int gm = m0 + m;
      Xs[m * (kKC + 1) + k] = (gm < M && k0 + k < p.d_in)
          ? ld_act(p.x, (int64_t)gm * p.d_in + k0 + k, p.act) : 0.f;
    }
    for (int i = threadIdx.x; i < D * kKC; i += kThreads) {
      const int n = i / kKC, k = i % kKC;
      Ws[n * (kKC + 1) + k] = k0 + k < p.d_in
          ? ld_act(p.w, ((int64_t)hh * D + n) * p.d_in + k0 + k, p.act) : 0.f;
    }
    __syncthreads();
    for (int k = 0; k < kKC; ++k) {
      const float wv = Ws[col * (kKC + 1) + k];
      for (int i = 0; i < rows_per; ++i)
        acc[i] += Xs[(rgi + i * rg) * (kKC + 1) + k] * wv;
    }
    __syncthreads();
  }
  // + (alpha/r) (x A^T) B^T
  if (r > 0) {
    const int64_t brow = (int64_t)head * D + col;
    for (int j = 0; j < r; ++j) {
      const float bv = ld_act(p.bm[proj], brow * r + j, p.act);
      for (int i = 0; i < rows_per; ++i) acc[i] += U[(rgi + i * rg) * 64 + j] * bv;
    }
  }
  for (int i = 0; i < rows_per; ++i) Y[(rgi + i * rg) * D + col] = acc[i];
  __syncthreads();
  // RoPE (rotate-half) on q and k; angle in fp64 for accuracy
  const bool rope = proj < 2 && p.rope_base > 0.f;
  const int H = proj == 0 ? p.Hq : p.Hkv;
  for (int i = threadIdx.x; i < kMT * D; i += kThreads) {
    const int m = i / D, d = i % D;
    const int gm = m0 + m;
    if (gm >= M) continue;
    const int b = gm / p.L, l = gm % p.L;
    float v = Y[i];
    if (rope) {
      const int half = D / 2, fi = d % half;
      float c, s;
      rope_cos_sin(p.pos0 + pos_of(p.pos_dev, p.pos_stride, b) + l, p.theta_hi[fi],
                   p.theta_lo[fi], &c, &s);
      if (d < half) v = Y[m * D + d] * c - Y[m * D + d + half] * s;
      else v = Y[m * D + d] * c + Y[m * D + d - half] * s;
    }
    st_act(p.out[proj], (((int64_t)b * H + head) * p.L + l) * D + d, v, p.act);
  }
}

// ---------------------------------------------------------------------------
// Few rows (M = B * L <= 16, the decode step): weight streaming.  Each warp
// owns one RoPE column pair (c, c + D/2) of one head and streams both weight
// rows with 16-byte loads; x (all M rows) sits in shared memory.  The
// rank-r branch: the CTA first forms (alpha/r) x A_p^T for its projection.
// ---------------------------------------------------------------------------
constexpr int kSkinnyWarps = 4;      // 3 CTAs per SM: one wave for up to 456 CTAs
constexpr int kSkinnyMaxM = 16;
constexpr int kSkinnyKIter = 8;      // 16-byte loads per row per lane in flight (2048 bf16)

template <typename T>
__device__ __forceinline__ void load8f(const T* p, float f[8]);
template <>
__device__ __forceinline__ void load8f<__nv_bfloat16>(const __nv_bfloat16* p, float f[8]) {
  uint4 u = __ldg(reinterpret_cast<const uint4*>(p));
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    float2 t = __bfloat1622float2(h[i]);
    f[2 * i] = t.x;
    f[2 * i + 1] = t.y;
  }
}
template <>
__device__ __forceinline__ void load8f<float>(const float* p, float f[8]) {
  float4 a = __ldg(reinterpret_cast<const float4*>(p));
  float4 b = __ldg(reinterpret_cast<const float4*>(p) + 1);
  f[0] = a.x; f[1] = a.y; f[2] = a.z; f[3] = a.w; f[4] = b.x; f[5] = b.y; f[6] = b.z; f[7] = b.w;
}

// Raw 8-element vector of activation type T (kept packed until used).
template <typename T> struct Raw8;
template <> struct Raw8<__nv_bfloat16> {
  uint4 u;
  __device__ __forceinline__ void load(const __nv_bfloat16* p) {
    u = __ldg(reinterpret_cast<const uint4*>(p));
  }
  __device__ __forceinline__ void to_float(float f[8]) const {
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      float2 t = __bfloat1622float2(h[i]);
      f[2 * i] = t.x;
      f[2 * i + 1] = t.y;
    }
  }
};
template <> struct Raw8<float> {
  float4 a, b;
  __device__ __forceinline__ void load(const float* p) {
    a = __ldg(reinterpret_cast<const float4*>(p));
    b = __ldg(reinterpret_cast<const float4*>(p) + 1);
  }
  __device__ __forceinline__ void to_float(float f[8]) const {
    f[0] = a.x; f[1] = a.y; f[2] = a.z; f[3] = a.w; f[4] = b.x; f[5] = b.y; f[6] = b.z; f[7] = b.w;
  }
};

template <typename T, int MM, int KITER>
__global__ void __launch_bounds__(kSkinnyWarps * 32, 3) project_skinny_kernel(ProjArgs p) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ float xsm[];             // [M][d_in] fp32, then U [M][64]
  const int M = p.B * p.L, D = p.D, K = p.d_in;
  const int half = D / 2;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int pairs_per_head = half;
  const int pair0 = blockIdx.x * kSkinnyWarps;      // CTA's first pair (stacked heads)
  const int hh = pair0 / pairs_per_head;           // all 8 pairs of a CTA share a head
  const int proj = hh < p.Hq ? 0 : hh < p.Hq + p.Hkv ? 1 : 2;
  const int head = proj == 0 ? hh : proj == 1 ? hh - p.Hq : hh - p.Hq - p.Hkv;
  const int r = p.r[proj];
  float* U = xsm + M * K;
  const T* x = reinterpret_cast<const T*>(p.x);
  const int c = (pair0 + warp) % pairs_per_head;    // channel within the first half
  const int n1 = hh * D + c, n2 = n1 + half;
  const T* W = reinterpret_cast<const T*>(p.w);
  const T* w1 = W + (int64_t)n1 * K;
  const T* w2 = W + (int64_t)n2 * K;
  // x -> shared memory (fp32): every thread issues all its loads, then stores
  {
    constexpr int XL = 8;                           // 16-byte loads per thread per round
    for (int base = threadIdx.x * 8; base < M * K; base += blockDim.x * 8 * XL) {
      Raw8<T> xv[XL];
#pragma unroll
      for (int u = 0; u < XL; ++u) {
        const int i = base + u * blockDim.x * 8;
        if (i < M * K) xv[u].load(x + i);
      }
#pragma unroll
      for (int u = 0; u < XL; ++u) {
        const int i = base + u * blockDim.x * 8;
        if (i < M * K) {
          float f[8];
          xv[u].to_float(f);
          *reinterpret_cast<float4*>(xsm + i) = make_float4(f[0], f[1], f[2], f[3]);
          *reinterpret_cast<float4*>(xsm + i + 4) = make_float4(f[4], f[5], f[6], f[7]);
        }
      }
    }
  }
  __syncthreads();
  // x A_p^T, one warp per rank: the row's 16-byte loads are all in flight
  // (passes of KITER x 256 channels), then M dot products reduced by shuffles.
  if (r > 0) {
    const T* A = reinterpret_cast<const T*>(p.a[proj]);
    for (int j = warp; j < r; j += kSkinnyWarps) {
      float acc[MM];
#pragma unroll
      for (int m = 0; m < MM; ++m) acc[m] = 0.f;
      for (int kp = 0; kp < K; kp += KITER * 256) {
        Raw8<T> av[KITER];
#pragma unroll
        for (int u = 0; u < KITER; ++u) {
          const int k = kp + lane * 8 + u * 256;
          if (k < K) av[u].load(A + (int64_t)j * K + k);
        }
#pragma unroll
        for (int u = 0; u < KITER; ++u) {
          const int k = kp + lane * 8 + u * 256;
          if (k < K) {
            float a[8];
            av[u].to_float(a);
#pragma unroll
            for (int m = 0; m < MM; ++m) {
              if (m < M) {
                const float4* xr4 = reinterpret_cast<const float4*>(xsm + m * K + k);
                const float4 xa = xr4[0], xb = xr4[1];
                acc[m] += a[0] * xa.x + a[1] * xa.y + a[2] * xa.z + a[3] * xa.w +
                          a[4] * xb.x + a[5] * xb.y + a[6] * xb.z + a[7] * xb.w;
              }
            }
          }
        }
      }
#pragma unroll
      for (int m = 0; m < MM; ++m) {
        float v = acc[m];
        for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        if (lane == 0 && m < M) U[m * 64 + j] = v;
      }
    }
  }
  // this warp's weight rows in passes of KITER x 256 channels: KITER 8-element
  // loads per row per lane in flight together (the bulk of the bytes)
  float acc1[MM], acc2[MM];
#pragma unroll
  for (int m = 0; m < MM; ++m) { acc1[m] = 0.f; acc2[m] = 0.f; }
  for (int kp = 0; kp < K; kp += KITER * 256) {
  Raw8<T> wa[KITER], wb[KITER];
#pragma unroll
  for (int u = 0; u < KITER; ++u) {
    const int k = kp + lane * 8 + u * 256;
    if (k < K) {
      wa[u].load(w1 + k);
      wb[u].load(w2 + k);
    }
  }
#pragma unroll
  for (int u = 0; u < KITER; ++u) {
    const int k = kp + lane * 8 + u * 256;
    if (k < K) {
      float a[8], bq[8];
      wa[u].to_float(a);
      wb[u].to_float(bq);
#pragma unroll
      for (int m = 0; m < MM; ++m) {
        if (m < M) {
          const float4* xr4 = reinterpret_cast<const float4*>(xsm + m * K + k);
          const float4 xa = xr4[0], xb = xr4[1];
          const float xr[8] = {xa.x, xa.y, xa.z, xa.w, xb.x, xb.y, xb.z, xb.w};
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            acc1[m] += a[e] * xr[e];
            acc2[m] += bq[e] * xr[e];
          }
        }
      }
    }
  }
  }
#pragma unroll
  for (int m = 0; m < MM; ++m) {
    for (int o = 16; o > 0; o >>= 1) {
      acc1[m] += __shfl_xor_sync(0xffffffffu, acc1[m], o);
      acc2[m] += __shfl_xor_sync(0xffffffffu, acc2[m], o);
    }
  }
  __syncthreads();                                  // U complete
  // rank-r up projection, RoPE, head-major store: lane m handles row m
  if (lane < M) {
    float y1 = 0.f, y2 = 0.f;
#pragma unroll
    for (int m = 0; m < MM; ++m)
      if (m == lane) { y1 = acc1[m]; y2 = acc2[m]; }
    if (r > 0) {
      const T* Bm = reinterpret_cast<const T*>(p.bm[proj]);
      const T* b1 = Bm + ((int64_t)head * D + c) * r;
      const T* b2 = Bm + ((int64_t)head * D + c + half) * r;
      for (int j0 = 0; j0 < r; j0 += 8) {          // r is a multiple of 8
        float f1[8], f2[8];
        load8f<T>(b1 + j0, f1);
        load8f<T>(b2 + j0, f2);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const float uu = U[lane * 64 + j0 + e] * p.alpha_over_r;
          y1 += uu * f1[e];
          y2 += uu * f2[e];
        }
      }
    }
    const int b = lane / p.L, l = lane % p.L;
    if (proj < 2 && p.rope_base > 0.f) {
      const int pos = p.pos0 + pos_of(p.pos_dev, p.pos_stride, b) + l;
      float cs, sn;
      rope_cos_sin(pos, p.theta_hi[c], p.theta_lo[c], &cs, &sn);
      const float o1 = y1 * cs - y2 * sn, o2 = y2 * cs + y1 * sn;
      y1 = o1;
      y2 = o2;
    }
    const int H = proj == 0 ? p.Hq : p.Hkv;
    const int64_t base = (((int64_t)b * H + head) * p.L + l) * D;
    st_act(p.out[proj], base + c, y1, p.act);
    st_act(p.out[proj], base + c + half, y2, p.act);
  }
}

template <int M16, int NT>
__global__ void __launch_bounds__(kDecWarps * 32) project_decode_mma_kernel(ProjArgs p) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ __align__(16) unsigned char dsm[];
  proj_decode_tile<M16, NT>(p, blockIdx.x, dsm);
}

template <int M16, int NT>
cudaError_t launch_decode_mma_nt(const ProjArgs& p, cudaStream_t s) {
  const size_t sm = proj_decode_smem_bytes(M16, NT, p.d_in);
  auto kern = project_decode_mma_kernel<M16, NT>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
  if (e != cudaSuccess) return e;
  const int tiles = (p.Hq + 2 * p.Hkv) * (p.D / 16);
  launch_pdl(kern, dim3(tiles), dim3(kDecWarps * 32), sm, s, p);
  return cudaGetLastError();
}

cudaError_t launch_decode_mma(const ProjArgs& p, cudaStream_t s) {
  const int M = p.B * p.L;
  const int rmax = max(p.r[0], max(p.r[1], p.r[2]));
  const int nt = 2 + rmax / 8;
  if (M <= 8) {
    if (nt <= 4) return launch_decode_mma_nt<8, 4>(p, s);
    return launch_decode_mma_nt<8, kDecMaxNt>(p, s);
  }
  if (nt <= 4) return launch_decode_mma_nt<16, 4>(p, s);
  return launch_decode_mma_nt<16, kDecMaxNt>(p, s);
}

template <typename T>
cudaError_t launch_skinny(const ProjArgs& p, cudaStream_t s) {
  const int M = p.B * p.L;
  const int pairs = (p.Hq + 2 * p.Hkv) * p.D / 2;
  const size_t sm = ((size_t)M * p.d_in + (size_t)kSkinnyMaxM * 64) * sizeof(float);
  // fp32 weights take twice the registers: half the loads per pass
  constexpr int KI = sizeof(T) == 2 ? kSkinnyKIter : kSkinnyKIter / 2;
  auto kern = M <= 4 ? project_skinny_kernel<T, 4, KI>
            : M <= 8 ? project_skinny_kernel<T, 8, KI> : project_skinny_kernel<T, kSkinnyMaxM, KI>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
  if (e != cudaSuccess) return e;
  launch_pdl(kern, dim3(pairs / kSkinnyWarps), dim3(kSkinnyWarps * 32), sm, s, p);
  return cudaGetLastError();
}

}  // namespace

// RoPE frequencies base^(-2i/D) for i < D/2 in fp64, split into hi + lo
// floats (zeros elsewhere, or everywhere when base = 0).
void rope_theta_table(float rope_base, int D, float* hi, float* lo) {
  for (int i = 0; i < 128; ++i) {
    const double th = i < D / 2 && rope_base > 0.f ? pow((double)rope_base, -2.0 * i / D) : 0.0;
    hi[i] = (float)th;
    lo[i] = (float)(th - (double)hi[i]);
  }
}

cudaError_t launch_project(const void* x, int B, int L, int d_in, const void* w,
                           const void* const a[3], const void* const bm[3], const int r[3],
                           float alpha_over_r, int Hq, int Hkv, int D, int pos0,
                           const int* pos_dev, float rope_base, int act,
                           void* const out[3], int* err, cudaStream_t s, int pos_stride) {
  ProjArgs p;
  p.x = x; p.w = w;
  for (int i = 0; i < 3; ++i) { p.a[i] = a[i]; p.bm[i] = bm[i]; p.r[i] = r[i]; p.out[i] = out[i]; }
  p.B = B; p.L = L; p.d_in = d_in; p.Hq = Hq; p.Hkv = Hkv; p.D = D; p.pos0 = pos0; p.act = act;
  p.pos_dev = pos_dev;
  p.pos_stride = pos_stride;
  p.alpha_over_r = alpha_over_r; p.rope_base = rope_base;
  rope_theta_table(rope_base, D, p.theta_hi, p.theta_lo);
  const int M = B * L;
  if (act == KVQ_BF16 && M > kSkinnyMaxM) {
    cudaError_t e = launch_project_tc(x, B, L, d_in, w, a, bm, r, alpha_over_r, Hq, Hkv, D, pos0,
                                      pos_dev, rope_base, out, err, s, nullptr, pos_stride);
    if (e != cudaErrorNotSupported) return e;
    (void)cudaGetLastError();
  }
  if (act == KVQ_BF16 && M <= 16 && d_in % 64 == 0) {
    cudaError_t e = launch_project_decode_stream(p, err, s);
    if (e != cudaErrorNotSupported) return e;
    (void)cudaGetLastError();
  }
  if (act == KVQ_BF16 && M <= 16 && d_in % 32 == 0 && (size_t)16 * d_in * 2 <= 160 * 1024)
    return launch_decode_mma(p, s);
  if (M <= kSkinnyMaxM && (size_t)M * d_in * 4 <= 120 * 1024 && d_in % 64 == 0)
    return act == KVQ_BF16 ? launch_skinny<__nv_bfloat16>(p, s) : launch_skinny<float>(p, s);
  const size_t sm = (size_t)(kMT * (kKC + 1) + 256 * (kKC + 1) + kMT * 64 + kMT * D) *
                    sizeof(float);
  cudaError_t e = cudaFuncSetAttribute(project_simt_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
  if (e != cudaSuccess) return e;
  dim3 grid((M + kMT - 1) / kMT, Hq + 2 * Hkv);
  launch_pdl(project_simt_kernel, dim3(grid), dim3(kThreads), sm, s, p);
  return cudaGetLastError();
}

}  // namespace kvq
