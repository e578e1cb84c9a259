// Backward of the packed path under the straight-through estimator
// (Section 3.3).  Newly appended states enter attention as
// x_hat + x - stopgrad(x): the forward sees the stored reconstruction and
// the gradient that reaches the keys and values, and through them the K and
// V adapters, is the gradient at the reconstruction, passed on unchanged.
// This is what lets the adapters train against the coded cache they will be
// served with (Sections 3.2-3.4).
//
// Attention, per (sequence, kv head) pair with its g = Hq / Hkv query heads
// stacked as M = g L rows (row m: head m / L, query m % L at position
// T - L + m % L):
//   S  = Q K^T                     P  = causal softmax(scale S) per row
//   dP = dO V^T                    dS = P o (dP - rowsum(P o dP)) scale
//   dQ = dS K                      dK = dS^T Q             dV = P^T dO
// K and V are the cache's reconstruction, materialised in fp32 in the
// caller's workspace with S (then P) and dP (then dS).
//
// Adapters (Eq. (1), Eq. (lora)): y_p = x W_p^T + (alpha/r) (x A_p^T) B_p^T,
// then RoPE on q and k.  With g_p the gradient of y_p (the output gradient
// rotated back), U_p = x A_p^T and V_p = g_p B_p:
//   dB_p = (alpha/r) g_p^T U_p      dA_p = (alpha/r) V_p^T x
//   dx   = g W + sum_p (alpha/r) V_p A_p
//
// Every product runs on one fp32 SIMT GEMM kernel with strided operands,
// batched over pairs and split over K where K is long and the output small.
#include <math.h>

#include "kvq_internal.cuh"
#include "proj_decode.cuh"
#include "reconstruct.cuh"

namespace kvq {
namespace {

// ---------------------------------------------------------------------------
// C[z] = alpha A[z] B[z] (+ C[z]) in fp32, A(m, k) and B(k, n) at strides.
// ---------------------------------------------------------------------------
constexpr int kBM = 64, kBN = 64, kBK = 16, kGemmThreads = 256;

enum MaskMode {
  kMaskNone = 0,
  kMaskRowsQueriesColsKeys = 1,   // m: stacked query rows, n: keys (S, dP)
  kMaskRowsQueriesKKeys = 2,      // m: stacked query rows, k: keys (dQ)
  kMaskRowsKeysKQueries = 3,      // m: keys, k: stacked query rows (dK, dV)
};

struct GemmArgs {
  const void* a;
  const void* b;
  float* c;
  int M, N, K;
  int64_t lda, ldb, ldc;      // A(m,k) = a[m lda + k] (K-major) or a[k lda + m]
  int64_t sa, sb, sc;         // batch strides in elements
  int batch, splits;          // grid.z = batch x splits; splits > 1 adds atomically
  float alpha;
  int accumulate;             // 1: C += alpha A B (splits > 1 implies it)
  int mask, L, T;             // causal structure of the attention products
};

// Latest key position visible to any of the stacked query rows [r0, r1).
__device__ __forceinline__ int max_visible(int r0, int r1, int L, int T) {
  const int last = r1 - 1;
  if (last / L != r0 / L) return T - 1;
  return T - L + last % L;
}

template <typename E>
__device__ __forceinline__ float ldf(const E* p, int64_t i);
template <>
__device__ __forceinline__ float ldf<float>(const float* p, int64_t i) { return p[i]; }
template <>
__device__ __forceinline__ float ldf<__nv_bfloat16>(const __nv_bfloat16* p, int64_t i) {
  return __bfloat162float(p[i]);
}

// Load one BK x 64 operand tile (rows r0.., k0..) into registers: 4 values per
// thread, consecutive threads on consecutive addresses of the contiguous axis.
template <typename E, bool KMAJOR>
__device__ __forceinline__ void load_tile(const E* p, int64_t ld, int r0, int R, int k0, int K,
                                          float v[4]) {
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int idx = threadIdx.x + kGemmThreads * i;
    int r, k;
    if (KMAJOR) { r = idx >> 4; k = idx & 15; } else { r = idx & 63; k = idx >> 6; }
    r += r0;
    k += k0;
    v[i] = (r < R && k < K) ? ldf<E>(p, KMAJOR ? (int64_t)r * ld + k : (int64_t)k * ld + r) : 0.f;
  }
}

template <bool KMAJOR>
__device__ __forceinline__ void store_tile(float (*s)[kBM + 4], const float v[4]) {
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int idx = threadIdx.x + kGemmThreads * i;
    int r, k;
    if (KMAJOR) { r = idx >> 4; k = idx & 15; } else { r = idx & 63; k = idx >> 6; }
    s[k][r] = v[i];
  }
}

// A_KMAJOR: A(m, k) = a[m lda + k], else a[k lda + m].
// B_KMAJOR: B(k, n) = b[n ldb + k], else b[k ldb + n].
template <typename TA, typename TB, bool A_KMAJOR, bool B_KMAJOR>
__global__ void __launch_bounds__(kGemmThreads) bgemm_kernel(GemmArgs g) {
  pdl_wait();
  __shared__ __align__(16) float As[2][kBK][kBM + 4];
  __shared__ __align__(16) float Bs[2][kBK][kBN + 4];
  const int z = blockIdx.z;
  const int bz = z / g.splits, sp = z % g.splits;
  const TA* A = reinterpret_cast<const TA*>(g.a) + (int64_t)bz * g.sa;
  const TB* Bp = reinterpret_cast<const TB*>(g.b) + (int64_t)bz * g.sb;
  float* C = g.c + (int64_t)bz * g.sc;
  const int m0 = blockIdx.y * kBM, n0 = blockIdx.x * kBN;

  // K range of this split, clipped by the causal structure.
  int kend = g.K;
  if (g.mask == kMaskRowsQueriesColsKeys &&
      n0 > max_visible(m0, min(m0 + kBM, g.M), g.L, g.T))
    return;                                    // every score of the tile is masked
  if (g.mask == kMaskRowsQueriesKKeys) kend = min(kend, max_visible(m0, min(m0 + kBM, g.M), g.L, g.T) + 1);
  const int ktiles = (kend + kBK - 1) / kBK;
  const int per = (ktiles + g.splits - 1) / g.splits;
  const int kt0 = sp * per, kt1 = min(ktiles, kt0 + per);
  if (kt0 >= kt1 && g.splits > 1) return;

  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  float acc[4][4] = {};
  float ra[4], rb[4];
  auto skip = [&](int kt) {
    return g.mask == kMaskRowsKeysKQueries &&
           max_visible(kt * kBK, min(kt * kBK + kBK, g.K), g.L, g.T) < m0;
  };
  int kt = kt0;
  while (kt < kt1 && skip(kt)) ++kt;
  if (kt < kt1) {
    load_tile<TA, A_KMAJOR>(A, g.lda, m0, g.M, kt * kBK, kend, ra);
    load_tile<TB, B_KMAJOR>(Bp, g.ldb, n0, g.N, kt * kBK, kend, rb);
  }
  int buf = 0;
  while (kt < kt1) {
    store_tile<A_KMAJOR>(As[buf], ra);
    store_tile<B_KMAJOR>(Bs[buf], rb);
    __syncthreads();
    int nxt = kt + 1;
    while (nxt < kt1 && skip(nxt)) ++nxt;
    if (nxt < kt1) {                           // prefetch the next tile into registers
      load_tile<TA, A_KMAJOR>(A, g.lda, m0, g.M, nxt * kBK, kend, ra);
      load_tile<TB, B_KMAJOR>(Bp, g.ldb, n0, g.N, nxt * kBK, kend, rb);
    }
#pragma unroll
    for (int k = 0; k < kBK; ++k) {
      const float4 av = *reinterpret_cast<const float4*>(&As[buf][k][ty * 4]);
      const float4 bv = *reinterpret_cast<const float4*>(&Bs[buf][k][tx * 4]);
      const float am[4] = {av.x, av.y, av.z, av.w};
      const float bn[4] = {bv.x, bv.y, bv.z, bv.w};
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(am[i], bn[j], acc[i][j]);
    }
    buf ^= 1;
    kt = nxt;
  }
  const bool atomic = g.splits > 1;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int m = m0 + ty * 4 + i;
    if (m >= g.M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + tx * 4 + j;
      if (n >= g.N) continue;
      float* dst = C + (int64_t)m * g.ldc + n;
      const float v = g.alpha * acc[i][j];
      if (atomic) atomicAdd(dst, v);
      else *dst = g.accumulate ? *dst + v : v;
    }
  }
}

template <typename TA, typename TB, bool AK, bool BK>
cudaError_t run_gemm(const GemmArgs& g, cudaStream_t s) {
  if (g.M <= 0 || g.N <= 0 || g.batch <= 0) return cudaSuccess;
  dim3 grid((g.N + kBN - 1) / kBN, (g.M + kBM - 1) / kBM, g.batch * g.splits);
  launch_pdl(bgemm_kernel<TA, TB, AK, BK>, grid, dim3(kGemmThreads), 0, s, g);
  return cudaGetLastError();
}

// Split K so that small outputs with long K still cover the SMs.
int choose_splits(int M, int N, int K, int batch) {
  const int64_t tiles = (int64_t)((M + kBM - 1) / kBM) * ((N + kBN - 1) / kBN) * batch;
  const int64_t want = 2LL * num_sms();
  if (tiles >= want) return 1;
  int s = (int)((want + tiles - 1) / tiles);
  const int maxs = max(1, K / (8 * kBK));      // keep at least 8 K tiles per split
  return max(1, min(s, min(maxs, 64)));
}

GemmArgs gemm_args(const void* a, int64_t lda, int64_t sa, const void* b, int64_t ldb,
                   int64_t sb, float* c, int64_t ldc, int64_t sc, int M, int N, int K,
                   int batch, float alpha) {
  GemmArgs g = {};
  g.a = a; g.b = b; g.c = c;
  g.M = M; g.N = N; g.K = K;
  g.lda = lda; g.ldb = ldb; g.ldc = ldc;
  g.sa = sa; g.sb = sb; g.sc = sc;
  g.batch = batch; g.splits = 1;
  g.alpha = alpha;
  return g;
}

// ---------------------------------------------------------------------------
// The reconstruction K_hat, V_hat [pairs][T][D] of pairs p0 .. p0 + npairs - 1
// (pair p = b Hkv + h) in fp32: one thread per 8 channels of a token.
// ---------------------------------------------------------------------------
__global__ void bwd_reconstruct_kernel(Geom g, int T, int p0, int npairs, float* kh, float* vh) {
  pdl_wait();
  const int c8 = g.D / 8;
  const int64_t n = (int64_t)npairs * T * c8;
  const int tq = g.fmt == KVQ_FMT_KIVI ? kivi_tq(T, g.R, g.G) : 0;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int c = (int)(i % c8);
    const int t = (int)((i / c8) % T);
    const int pp = (int)(i / ((int64_t)c8 * T));
    const int b = (p0 + pp) / g.H, h = (p0 + pp) % g.H;
    float* dst[2] = {kh + ((int64_t)pp * T + t) * g.D + 8 * c,
                     vh + ((int64_t)pp * T + t) * g.D + 8 * c};
    const bool raw = g.fmt == KVQ_FMT_FLOAT || (g.fmt == KVQ_FMT_KIVI && t >= tq);
    for (int which = 0; which < 2; ++which) {
      float v[8];
      if (raw && g.act == KVQ_F32) {
        const int slot = g.fmt == KVQ_FMT_KIVI ? t % g.ring : t;
        const float* src = plane_ptr<float>(g, which ? KVQ_PLANE_V_FULL : KVQ_PLANE_K_FULL, b, h,
                                            slot, 8 * c);
#pragma unroll
        for (int e = 0; e < 8; ++e) v[e] = src[e];
      } else {
        deq8(g, which, b, h, t, c, T, tq, v);
      }
#pragma unroll
      for (int e = 0; e < 8; e += 4)
        *reinterpret_cast<float4*>(dst[which] + e) = make_float4(v[e], v[e + 1], v[e + 2], v[e + 3]);
    }
  }
}

// ---------------------------------------------------------------------------
// Per stacked query row: P = causal softmax(scale S) over S, and
// dS = P o (dP - sum_n P dP) scale over dP; masked entries become 0.
// One CTA of 256 threads per row, rows of all pairs of the chunk.
// ---------------------------------------------------------------------------
constexpr int kRowThreads = 256;

__device__ __forceinline__ float block_reduce(float v, bool is_max, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float w = __shfl_xor_sync(0xffffffffu, v, o);
    v = is_max ? fmaxf(v, w) : v + w;
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();                          // red[] free from the previous reduction
  if (lane == 0) red[warp] = v;
  __syncthreads();
  v = red[lane < kRowThreads / 32 ? lane : 0];
#pragma unroll
  for (int o = 4; o > 0; o >>= 1) {
    const float w = __shfl_xor_sync(0xffffffffu, v, o);
    v = is_max ? fmaxf(v, w) : v + w;
  }
  return __shfl_sync(0xffffffffu, v, 0);   // lanes 0-7 hold the total
}

__global__ void __launch_bounds__(kRowThreads)
bwd_softmax_ds_kernel(float* S, float* dP, int M, int T, int L, float scale) {
  pdl_wait();
  __shared__ float red[kRowThreads / 32];
  const int m = blockIdx.x;
  const int64_t row = ((int64_t)blockIdx.y * M + m) * T;
  float* s = S + row;
  float* dp = dP + row;
  const int nvis = T - L + m % L + 1;        // keys 0 .. T - L + l are visible
  float mx = -INFINITY;
  for (int n = threadIdx.x; n < nvis; n += kRowThreads) mx = fmaxf(mx, s[n]);
  mx = block_reduce(mx, true, red);
  float sum = 0.f, dot = 0.f;
  for (int n = threadIdx.x; n < nvis; n += kRowThreads) {
    const float e = expf(scale * (s[n] - mx));
    sum += e;
    dot = fmaf(e, dp[n], dot);
  }
  sum = block_reduce(sum, false, red);
  dot = block_reduce(dot, false, red);
  const float inv = 1.f / sum;
  const float delta = dot * inv;             // sum_n P dP
  for (int n = threadIdx.x; n < T; n += kRowThreads) {
    float p = 0.f, ds = 0.f;
    if (n < nvis) {
      p = expf(scale * (s[n] - mx)) * inv;
      ds = p * (dp[n] - delta) * scale;
    }
    s[n] = p;
    dp[n] = ds;
  }
}

// ---------------------------------------------------------------------------
// Adapter backward: G [B L][(Hq + 2 Hkv) D], the gradient of the projection
// before RoPE (columns in w_qkv's row order).  d_k and d_v hold kv_rows
// tokens per (sequence, head), of which the last L are the tokens of x.
// ---------------------------------------------------------------------------
struct GatherArgs {
  const float* dq;
  const float* dk;
  const float* dv;
  float* G;
  int B, L, Hq, Hkv, D, kv_rows, pos0;
  float theta_hi[128], theta_lo[128];
};

__global__ void lora_gather_kernel(GatherArgs a) {
  pdl_wait();
  const int half = a.D / 2;
  const int heads = a.Hq + 2 * a.Hkv;
  const int64_t ntot = (int64_t)heads * a.D;
  const int64_t n = (int64_t)a.B * a.L * heads * half;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int c = (int)(i % half);
    const int hh = (int)((i / half) % heads);
    const int64_t bl = i / ((int64_t)half * heads);
    const int b = (int)(bl / a.L), l = (int)(bl % a.L);
    const float* src;
    bool rope = true;
    if (hh < a.Hq) {
      src = a.dq + (((int64_t)b * a.Hq + hh) * a.L + l) * a.D;
    } else {
      const int h = (hh - a.Hq) % a.Hkv;
      const bool isv = hh >= a.Hq + a.Hkv;
      src = (isv ? a.dv : a.dk) +
            (((int64_t)b * a.Hkv + h) * a.kv_rows + (a.kv_rows - a.L + l)) * a.D;
      rope = !isv;
    }
    float g1 = src[c], g2 = src[c + half];
    if (rope && a.theta_hi[0] != 0.f) {       // the rotation transposed: angle -pos theta
      float cs, sn;
      pdec::rope_cos_sin(a.pos0 + l, a.theta_hi[c], a.theta_lo[c], &cs, &sn);
      const float r1 = fmaf(g1, cs, g2 * sn);
      const float r2 = fmaf(g2, cs, -g1 * sn);
      g1 = r1;
      g2 = r2;
    }
    float* dst = a.G + bl * ntot + (int64_t)hh * a.D;
    dst[c] = g1;
    dst[c + half] = g2;
  }
}

// Rows of G [rows][n] fp32, in place, as [rows][2n] bf16: the high parts
// (g rounded to bf16) then the bf16 of the remainders, so that the two halves
// carry about 16 significant bits of g for a bf16 tensor-core product.  One
// CTA per row at a time: the row goes through shared memory first.
__global__ void __launch_bounds__(256) bwd_split_rows_kernel(float* G, int rows, int n) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ float rowbuf[];
  for (int r = blockIdx.x; r < rows; r += gridDim.x) {
    float* g = G + (int64_t)r * n;
    for (int j = threadIdx.x; j < n; j += blockDim.x) rowbuf[j] = g[j];
    __syncthreads();
    __nv_bfloat16* o = reinterpret_cast<__nv_bfloat16*>(g);
    for (int j = threadIdx.x; j < n; j += blockDim.x) {
      const float v = rowbuf[j];
      const __nv_bfloat16 hi = __float2bfloat16_rn(v);
      o[j] = hi;
      o[n + j] = __float2bfloat16_rn(v - __bfloat162float(hi));
    }
    __syncthreads();
  }
}

// Wt [d][n] = W [n][d] (bf16), 32 x 32 tiles through shared memory.
__global__ void __launch_bounds__(256) bwd_transpose_kernel(const __nv_bfloat16* __restrict__ W,
                                                            __nv_bfloat16* __restrict__ Wt, int n,
                                                            int d) {
  pdl_wait();
  pdl_trigger();
  __shared__ __nv_bfloat16 tile[32][33];
  const int n0 = blockIdx.y * 32, d0 = blockIdx.x * 32;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;   // 8 rows per pass
  for (int i = ty; i < 32; i += 8)
    if (n0 + i < n && d0 + tx < d) tile[i][tx] = W[(int64_t)(n0 + i) * d + d0 + tx];
  __syncthreads();
  for (int i = ty; i < 32; i += 8)
    if (d0 + i < d && n0 + tx < n) Wt[(int64_t)(d0 + i) * n + n0 + tx] = tile[tx][i];
}

int grid_for(int64_t n, int threads) {
  const int64_t blocks = (n + threads - 1) / threads;
  return (int)std::min<int64_t>(blocks, (int64_t)num_sms() * 16);
}

}  // namespace

// ---------------------------------------------------------------------------
// Host side.
// ---------------------------------------------------------------------------
namespace {

// run_gemm with the activation-typed operand(s) chosen by `act`.
template <bool AK, bool BK>
cudaError_t gemm_act_b(const GemmArgs& g, int act, cudaStream_t s) {   // B in act dtype
  return act == KVQ_BF16 ? run_gemm<float, __nv_bfloat16, AK, BK>(g, s)
                         : run_gemm<float, float, AK, BK>(g, s);
}
template <bool AK, bool BK>
cudaError_t gemm_act_a(const GemmArgs& g, int act, cudaStream_t s) {   // A in act dtype
  return act == KVQ_BF16 ? run_gemm<__nv_bfloat16, float, AK, BK>(g, s)
                         : run_gemm<float, float, AK, BK>(g, s);
}
template <bool AK, bool BK>
cudaError_t gemm_act_ab(const GemmArgs& g, int act, cudaStream_t s) {  // both in act dtype
  return act == KVQ_BF16 ? run_gemm<__nv_bfloat16, __nv_bfloat16, AK, BK>(g, s)
                         : run_gemm<float, float, AK, BK>(g, s);
}

size_t a256(size_t x) { return (x + 255) & ~size_t(255); }

}  // namespace

size_t attend_backward_pair_bytes(const Geom& g, int T, int L) {
  const size_t gl = (size_t)(g.Hq / g.H) * L;
  return a256((2 * (size_t)T * g.D + 2 * gl * T) * sizeof(float));
}

cudaError_t launch_attend_backward(const Geom& g, int T, const void* q, const void* d_out,
                                   int L, float scale, float* dq, float* dk, float* dv,
                                   void* ws, size_t ws_bytes, cudaStream_t s) {
  const int pairs = g.B * g.H, grp = g.Hq / g.H, D = g.D;
  const int M = grp * L;
  const int act = g.act;
  const size_t esz = act == KVQ_BF16 ? 2 : 4;
  const int chunk = (int)std::min<size_t>(pairs, ws_bytes / attend_backward_pair_bytes(g, T, L));
  cudaError_t e = cudaSuccess;
  for (int p0 = 0; p0 < pairs && e == cudaSuccess; p0 += chunk) {
    const int np = std::min(chunk, pairs - p0);
    float* kh = static_cast<float*>(ws);
    float* vh = kh + (size_t)np * T * D;
    float* S = vh + (size_t)np * T * D;
    float* dP = S + (size_t)np * M * T;
    const char* qp = static_cast<const char*>(q) + (size_t)p0 * M * D * esz;
    const char* op = static_cast<const char*>(d_out) + (size_t)p0 * M * D * esz;
    launch_pdl(bwd_reconstruct_kernel, dim3(grid_for((int64_t)np * T * D / 8, 256)), dim3(256),
               0, s, g, T, p0, np, kh, vh);
    e = cudaGetLastError();
    // S = Q K^T and dP = dO V^T (tiles above the causal edge skipped)
    GemmArgs ga = gemm_args(qp, D, (int64_t)M * D, kh, D, (int64_t)T * D, S, T, (int64_t)M * T,
                            M, T, D, np, 1.f);
    ga.mask = kMaskRowsQueriesColsKeys; ga.L = L; ga.T = T;
    if (e == cudaSuccess) e = gemm_act_a<true, true>(ga, act, s);
    ga.a = op; ga.b = vh; ga.c = dP;
    if (e == cudaSuccess) e = gemm_act_a<true, true>(ga, act, s);
    if (e == cudaSuccess) {
      launch_pdl(bwd_softmax_ds_kernel, dim3(M, np), dim3(kRowThreads), 0, s, S, dP, M, T, L,
                 scale);
      e = cudaGetLastError();
    }
    // dQ = dS K
    GemmArgs gq = gemm_args(dP, T, (int64_t)M * T, kh, D, (int64_t)T * D,
                            dq + (size_t)p0 * M * D, D, (int64_t)M * D, M, D, T, np, 1.f);
    gq.mask = kMaskRowsQueriesKKeys; gq.L = L; gq.T = T;
    if (e == cudaSuccess) e = run_gemm<float, float, true, false>(gq, s);
    // dK = dS^T Q and dV = P^T dO
    GemmArgs gk = gemm_args(dP, T, (int64_t)M * T, qp, D, (int64_t)M * D,
                            dk + (size_t)p0 * T * D, D, (int64_t)T * D, T, D, M, np, 1.f);
    gk.mask = kMaskRowsKeysKQueries; gk.L = L; gk.T = T;
    if (e == cudaSuccess) e = gemm_act_b<false, false>(gk, act, s);
    gk.a = S; gk.b = op; gk.c = dv + (size_t)p0 * T * D;
    if (e == cudaSuccess) e = gemm_act_b<false, false>(gk, act, s);
  }
  return e;
}

size_t lora_backward_bytes(int B, int L, int d_in, int Hq, int Hkv, int D, const int r[3]) {
  const size_t BL = (size_t)B * L;
  size_t n = a256(BL * (Hq + 2 * Hkv) * D * sizeof(float));
  for (int p = 0; p < 3; ++p) n += 2 * a256(BL * r[p] * sizeof(float));
  n += a256((size_t)d_in * (Hq + 2 * Hkv) * D * 2);   // W^T in bf16 for the d_x product
  return n;
}

// d_x on tcgen05 needs bf16 activations and whole 64-element K slices and
// 128-column output tiles.
static bool dx_on_tc(int act, int d_in, int ntot) {
  return act == KVQ_BF16 && d_in % 128 == 0 && ntot % 64 == 0;
}

cudaError_t launch_lora_backward(const void* x, int B, int L, int d_in, const void* w,
                                 const void* const a[3], const void* const bm[3],
                                 const int r[3], float alpha_over_r, int Hq, int Hkv, int D,
                                 int pos0, float rope_base, int act, const float* dq,
                                 const float* dk, const float* dv, int kv_rows,
                                 float* const da[3], float* const db[3], float* dx, void* ws,
                                 cudaStream_t s) {
  const int BL = B * L;
  const int ntot = (Hq + 2 * Hkv) * D;
  const int nout[3] = {Hq * D, Hkv * D, Hkv * D};
  const int off[3] = {0, Hq * D, (Hq + Hkv) * D};
  char* wp = static_cast<char*>(ws);
  float* G = reinterpret_cast<float*>(wp);
  wp += a256((size_t)BL * ntot * sizeof(float));
  float* U[3];
  float* V[3];
  for (int p = 0; p < 3; ++p) {
    U[p] = reinterpret_cast<float*>(wp);
    wp += a256((size_t)BL * r[p] * sizeof(float));
    V[p] = reinterpret_cast<float*>(wp);
    wp += a256((size_t)BL * r[p] * sizeof(float));
  }
  __nv_bfloat16* Wt = reinterpret_cast<__nv_bfloat16*>(wp);   // [d_in][ntot]
  GatherArgs ga;
  ga.dq = dq; ga.dk = dk; ga.dv = dv; ga.G = G;
  ga.B = B; ga.L = L; ga.Hq = Hq; ga.Hkv = Hkv; ga.D = D; ga.kv_rows = kv_rows; ga.pos0 = pos0;
  rope_theta_table(rope_base, D, ga.theta_hi, ga.theta_lo);
  launch_pdl(lora_gather_kernel, dim3(grid_for((int64_t)BL * (Hq + 2 * Hkv) * D / 2, 256)),
             dim3(256), 0, s, ga);
  cudaError_t e = cudaGetLastError();
  for (int p = 0; p < 3 && e == cudaSuccess; ++p) {
    if (r[p] == 0) continue;
    // U_p = x A_p^T  [BL][r] and V_p = g_p B_p  [BL][r]: narrow outputs over
    // long K, split over K (accumulated atomically into zeroed outputs)
    GemmArgs gu = gemm_args(x, d_in, 0, a[p], d_in, 0, U[p], r[p], 0, BL, r[p], d_in, 1, 1.f);
    gu.splits = choose_splits(BL, r[p], d_in, 1);
    if (gu.splits > 1) e = cudaMemsetAsync(U[p], 0, (size_t)BL * r[p] * sizeof(float), s);
    if (e == cudaSuccess) e = gemm_act_ab<true, true>(gu, act, s);
    GemmArgs gv = gemm_args(G + off[p], ntot, 0, bm[p], r[p], 0, V[p], r[p], 0, BL, r[p],
                            nout[p], 1, 1.f);
    gv.splits = choose_splits(BL, r[p], nout[p], 1);
    if (e == cudaSuccess && gv.splits > 1)
      e = cudaMemsetAsync(V[p], 0, (size_t)BL * r[p] * sizeof(float), s);
    if (e == cudaSuccess) e = gemm_act_b<true, false>(gv, act, s);
    // dB_p = (alpha/r) g_p^T U_p  [n_p][r], split over the BL rows
    GemmArgs gb = gemm_args(G + off[p], ntot, 0, U[p], r[p], 0, db[p], r[p], 0, nout[p], r[p],
                            BL, 1, alpha_over_r);
    gb.splits = choose_splits(nout[p], r[p], BL, 1);
    if (e == cudaSuccess && gb.splits > 1)
      e = cudaMemsetAsync(db[p], 0, (size_t)nout[p] * r[p] * sizeof(float), s);
    if (e == cudaSuccess) e = run_gemm<float, float, false, false>(gb, s);
    // dA_p = (alpha/r) V_p^T x  [r][d_in]
    GemmArgs gA = gemm_args(V[p], r[p], 0, x, d_in, 0, da[p], d_in, 0, r[p], d_in, BL, 1,
                            alpha_over_r);
    gA.splits = choose_splits(r[p], d_in, BL, 1);
    if (e == cudaSuccess && gA.splits > 1)
      e = cudaMemsetAsync(da[p], 0, (size_t)r[p] * d_in * sizeof(float), s);
    if (e == cudaSuccess) e = gemm_act_b<false, false>(gA, act, s);
  }
  if (dx && e == cudaSuccess) {
    // dx = g W + sum_p (alpha/r) V_p A_p
    if (dx_on_tc(act, d_in, ntot)) {
      // g W on tcgen05: g split into bf16 high and low parts in place (G is
      // not read again), [g_hi | g_lo] times [W^T | W^T] along K
      int* err = device_error_word();
      if (!err) return cudaErrorInvalidDevice;
      launch_pdl(bwd_transpose_kernel, dim3((d_in + 31) / 32, (ntot + 31) / 32), dim3(256), 0, s,
                 reinterpret_cast<const __nv_bfloat16*>(w), Wt, ntot, d_in);
      e = cudaGetLastError();
      const size_t sm = (size_t)ntot * sizeof(float);
      if (e == cudaSuccess && sm > 48 * 1024)
        e = cudaFuncSetAttribute(bwd_split_rows_kernel,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
      if (e == cudaSuccess) {
        launch_pdl(bwd_split_rows_kernel, dim3(std::min(BL, num_sms() * 8)), dim3(256), sm, s, G,
                   BL, ntot);
        e = cudaGetLastError();
      }
      if (e == cudaSuccess) e = launch_gemm_tc_bf16(G, BL, 2 * ntot, Wt, d_in, ntot, dx, err, s);
    } else {
      GemmArgs gx = gemm_args(G, ntot, 0, w, d_in, 0, dx, d_in, 0, BL, d_in, ntot, 1, 1.f);
      e = gemm_act_b<true, false>(gx, act, s);
    }
    for (int p = 0; p < 3 && e == cudaSuccess; ++p) {
      if (r[p] == 0) continue;
      GemmArgs gl = gemm_args(V[p], r[p], 0, a[p], d_in, 0, dx, d_in, 0, BL, d_in, r[p], 1,
                              alpha_over_r);
      gl.accumulate = 1;
      e = gemm_act_b<true, false>(gl, act, s);
    }
  }
  return e;
}

}  // namespace kvq
