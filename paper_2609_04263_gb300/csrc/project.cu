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
  const int* pos_dev;   // if set, positions start at *pos_dev + pos0
  float alpha_over_r, rope_base;
  // RoPE frequencies base^(-2i/D), i < D/2, computed in fp64 on the host and
  // split into hi + lo floats
  float theta_hi[128], theta_lo[128];
};

// cos and sin of pos * theta in fp32 to about 1e-7 absolute for positions
// below 2^24: pos * theta_hi is formed exactly as p + e (FMA), reduced by
// 2 pi in three parts (the first exact for multiples below 2^15), then the
// small remainder goes to sincosf.
__device__ __forceinline__ void rope_cos_sin(int pos, float th_hi, float th_lo, float* c,
                                             float* s) {
  const float x = (float)pos;
  const float p = x * th_hi;
  const float e = fmaf(x, th_hi, -p) + x * th_lo;
  const float k = rintf(p * 0.15915494309189535f);          // 1 / (2 pi)
  float r = fmaf(-k, 6.28125f, p);                            // 2 pi = 6.28125
  r = fmaf(-k, 1.9353071795864769e-3f, r);                    //   + 1.9353072e-3
  r = fmaf(-k, 1.0253132e-11f, r);                            //   + 1.0253e-11 (remainder)
  r += e;
  sincosf(r, s, c);
}

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
  const int pos_base = p.pos0 + (p.pos_dev ? *p.pos_dev : 0);
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
      rope_cos_sin(pos_base + l, p.theta_hi[fi], p.theta_lo[fi], &c, &s);
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
constexpr int kSkinnyWarps = 8;
constexpr int kSkinnyMaxM = 16;

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

template <typename T, int MM>
__global__ void __launch_bounds__(kSkinnyWarps * 32) project_skinny_kernel(ProjArgs p) {
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
  for (int i = threadIdx.x * 8; i < M * K; i += blockDim.x * 8) {
    float f[8];
    load8f<T>(x + i, f);
#pragma unroll
    for (int j = 0; j < 8; ++j) xsm[i + j] = f[j];
  }
  __syncthreads();
  // (alpha/r) x A_p^T: warp w takes ranks w, w + 8, ...
  if (r > 0) {
    const T* A = reinterpret_cast<const T*>(p.a[proj]);
    for (int j = warp; j < r; j += kSkinnyWarps) {
      float acc[MM];
#pragma unroll
      for (int m = 0; m < MM; ++m) acc[m] = 0.f;
      for (int k = lane * 8; k < K; k += 256) {
        float a[8];
        load8f<T>(A + (int64_t)j * K + k, a);
#pragma unroll
        for (int m = 0; m < MM; ++m) {
          if (m < M) {
            const float* xr = xsm + m * K + k;
#pragma unroll
            for (int e = 0; e < 8; ++e) acc[m] += a[e] * xr[e];
          }
        }
      }
#pragma unroll
      for (int m = 0; m < MM; ++m) {
        float v = acc[m];
        for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        if (lane == 0 && m < M) U[m * 64 + j] = v * p.alpha_over_r;
      }
    }
  }
  __syncthreads();
  const int c = (pair0 + warp) % pairs_per_head;    // channel within the first half
  const int n1 = hh * D + c, n2 = n1 + half;
  const T* W = reinterpret_cast<const T*>(p.w);
  const T* w1 = W + (int64_t)n1 * K;
  const T* w2 = W + (int64_t)n2 * K;
  float acc1[MM], acc2[MM];
#pragma unroll
  for (int m = 0; m < MM; ++m) { acc1[m] = 0.f; acc2[m] = 0.f; }
  constexpr int kUnroll = 4;
  for (int k0 = lane * 8; k0 < K; k0 += 256 * kUnroll) {
    float a[kUnroll][8], b[kUnroll][8];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int k = k0 + u * 256;
      if (k < K) {
        load8f<T>(w1 + k, a[u]);
        load8f<T>(w2 + k, b[u]);
      }
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int k = k0 + u * 256;
      if (k < K) {
#pragma unroll
        for (int m = 0; m < MM; ++m) {
          if (m < M) {
            const float4* xr4 = reinterpret_cast<const float4*>(xsm + m * K + k);
            const float4 xa = xr4[0], xb = xr4[1];
            const float xr[8] = {xa.x, xa.y, xa.z, xa.w, xb.x, xb.y, xb.z, xb.w};
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              acc1[m] += a[u][e] * xr[e];
              acc2[m] += b[u][e] * xr[e];
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
  // rank-r up projection, RoPE, head-major store: lane m handles row m
  if (lane < M) {
    float y1 = 0.f, y2 = 0.f;
#pragma unroll
    for (int m = 0; m < MM; ++m)
      if (m == lane) { y1 = acc1[m]; y2 = acc2[m]; }
    if (r > 0) {
      const T* Bm = reinterpret_cast<const T*>(p.bm[proj]);
      const int64_t b1 = ((int64_t)head * D + c) * r, b2 = ((int64_t)head * D + c + half) * r;
      for (int j = 0; j < r; ++j) {
        const float u = U[lane * 64 + j];
        y1 += u * ld_act(Bm, b1 + j, p.act);
        y2 += u * ld_act(Bm, b2 + j, p.act);
      }
    }
    const int b = lane / p.L, l = lane % p.L;
    if (proj < 2 && p.rope_base > 0.f) {
      const int pos = p.pos0 + (p.pos_dev ? *p.pos_dev : 0) + l;
      float cs, sn;
      rope_cos_sin(pos, p.theta_hi[c], p.theta_lo[c], &cs, &sn);
      const float o1 = y1 * cs - y2 * sn, o2 = y2 * cs + y1 * sn;
      y1 = o1;
      y2 = o2;
    }
    const int H = proj == 0 ? p.Hq : proj == 1 ? p.Hkv : p.Hkv;
    const int64_t base = (((int64_t)b * H + head) * p.L + l) * D;
    st_act(p.out[proj], base + c, y1, p.act);
    st_act(p.out[proj], base + c + half, y2, p.act);
  }
}

template <typename T>
cudaError_t launch_skinny(const ProjArgs& p, cudaStream_t s) {
  const int M = p.B * p.L;
  const int pairs = (p.Hq + 2 * p.Hkv) * p.D / 2;
  const size_t sm = ((size_t)M * p.d_in + (size_t)M * 64) * sizeof(float);
  auto kern = M <= 4 ? project_skinny_kernel<T, 4> : project_skinny_kernel<T, kSkinnyMaxM>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
  if (e != cudaSuccess) return e;
  kern<<<pairs / kSkinnyWarps, kSkinnyWarps * 32, sm, s>>>(p);
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
                           void* const out[3], int* err, cudaStream_t s) {
  ProjArgs p;
  p.x = x; p.w = w;
  for (int i = 0; i < 3; ++i) { p.a[i] = a[i]; p.bm[i] = bm[i]; p.r[i] = r[i]; p.out[i] = out[i]; }
  p.B = B; p.L = L; p.d_in = d_in; p.Hq = Hq; p.Hkv = Hkv; p.D = D; p.pos0 = pos0; p.act = act;
  p.pos_dev = pos_dev;
  p.alpha_over_r = alpha_over_r; p.rope_base = rope_base;
  rope_theta_table(rope_base, D, p.theta_hi, p.theta_lo);
  const int M = B * L;
  if (act == KVQ_BF16 && M > kSkinnyMaxM) {
    cudaError_t e = launch_project_tc(x, B, L, d_in, w, a, bm, r, alpha_over_r, Hq, Hkv, D, pos0,
                                      pos_dev, rope_base, out, err, s);
    if (e != cudaErrorNotSupported) return e;
    (void)cudaGetLastError();
  }
  if (M <= kSkinnyMaxM && (size_t)M * d_in * 4 <= 160 * 1024 && d_in % 8 == 0)
    return act == KVQ_BF16 ? launch_skinny<__nv_bfloat16>(p, s) : launch_skinny<float>(p, s);
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
