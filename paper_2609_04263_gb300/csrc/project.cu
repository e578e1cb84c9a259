// LoRA-adapted Q/K/V projection (Section 3, Eq. 1 and Eq. lora) with rotary
// positions, written head-major.  The adapter stays an explicit rank-r
// branch (Section 3.4): y = x W^T + (alpha/r) (x A^T) B^T.
#include <math.h>

#include "kvq_internal.cuh"

namespace kvq {
namespace {

constexpr int kMT = 32;     // rows per CTA
constexpr int kKC = 32;     // k chunk
constexpr int kThreads = 256;

struct ProjArgs {
  const void* x;
  const void* w;
  const void* a[3];
  const void* bm[3];
  int r[3];
  void* out[3];
  int B, L, d_in, Hq, Hkv, D, pos0, act;
  float alpha_over_r, rope_base;
};

// One CTA: kMT rows of x times one head's D output columns.
__global__ void __launch_bounds__(kThreads) project_simt_kernel(ProjArgs p) {
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
      const double theta = pow((double)p.rope_base, -2.0 * fi / D);
      const double ang = (double)(p.pos0 + l) * theta;
      const float c = (float)cos(ang), s = (float)sin(ang);
      if (d < half) v = Y[m * D + d] * c - Y[m * D + d + half] * s;
      else v = Y[m * D + d] * c + Y[m * D + d - half] * s;
    }
    st_act(p.out[proj], (((int64_t)b * H + head) * p.L + l) * D + d, v, p.act);
  }
}

}  // namespace

cudaError_t launch_project(const void* x, int B, int L, int d_in, const void* w,
                           const void* const a[3], const void* const bm[3], const int r[3],
                           float alpha_over_r, int Hq, int Hkv, int D, int pos0,
                           float rope_base, int act, void* const out[3], int* err,
                           cudaStream_t s) {
  (void)err;
  ProjArgs p;
  p.x = x; p.w = w;
  for (int i = 0; i < 3; ++i) { p.a[i] = a[i]; p.bm[i] = bm[i]; p.r[i] = r[i]; p.out[i] = out[i]; }
  p.B = B; p.L = L; p.d_in = d_in; p.Hq = Hq; p.Hkv = Hkv; p.D = D; p.pos0 = pos0; p.act = act;
  p.alpha_over_r = alpha_over_r; p.rope_base = rope_base;
  const int M = B * L;
  const size_t sm = (size_t)(kMT * (kKC + 1) + 256 * (kKC + 1) + kMT * 64 + kMT * D) *
                    sizeof(float);
  cudaError_t e = cudaFuncSetAttribute(project_simt_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
  if (e != cudaSuccess) return e;
  dim3 grid((M + kMT - 1) / kMT, Hq + 2 * Hkv);
  project_simt_kernel<<<grid, kThreads, sm, s>>>(p);
  return cudaGetLastError();
}

}  // namespace kvq
