// Attention over the stored reconstruction R_phi(K, V) (Sections 3.2-3.3).
// Prefill: causal attention of the newest L queries over all T tokens.
// Decode: L = 1, split over the tokens, partials merged by log-sum-exp.
#include <math.h>

#include "kvq_internal.cuh"

namespace kvq {
namespace {

constexpr int kTile = 32;       // tokens per shared-memory tile
constexpr int kThreads = 128;

// Split-K partials of (b, q head): kMaxSplits rows of (m, l, o[D]).
__device__ __forceinline__ float* ws_row(const Geom& g, int b, int hq) {
  return reinterpret_cast<float*>(g.pl[KVQ_PLANE_WORKSPACE].p) +
         ((int64_t)b * g.Hq + hq) * kMaxSplits * (g.D + kWsStride);
}

__device__ __forceinline__ unsigned code_at(const uint8_t* row, int d, int bits) {
  const int bit = d * bits;
  return (row[bit >> 3] >> (bit & 7)) & ((1u << bits) - 1);
}

// Reconstruct tokens [t0, t0 + n) of one (b, h) into dst [n][ld] (fp32).
// which = 0 keys, 1 values.  T = tokens stored.
__device__ void dequant_tile(const Geom& g, int which, int b, int h, int t0, int n, int T,
                             float* dst, int ld, float inv_sqrt_d) {
  const int D = g.D, G = g.G;
  const int bits = which ? g.vb : g.kb;
  const int P_CODES = which ? KVQ_PLANE_V_CODES : KVQ_PLANE_K_CODES;
  const int P_SCALE = which ? KVQ_PLANE_V_SCALE : KVQ_PLANE_K_SCALE;
  const int P_ZERO = which ? KVQ_PLANE_V_ZERO : KVQ_PLANE_K_ZERO;
  const int P_FULL = which ? KVQ_PLANE_V_FULL : KVQ_PLANE_K_FULL;
  const int P_PEND = which ? KVQ_PLANE_V_PEND : KVQ_PLANE_K_PEND;
  const int P_ROW = which ? KVQ_PLANE_V_ROW : KVQ_PLANE_K_ROW;
  const int P_COL = which ? KVQ_PLANE_V_COL : KVQ_PLANE_K_COL;
  const int tq = g.fmt == KVQ_FMT_KIVI ? kivi_tq(T, g.R, G) : 0;
  const int nbq = g.fmt == KVQ_FMT_KVARN ? kvarn_nblocks(T, g.S, G) * G : 0;
  for (int i = threadIdx.x; i < n * D; i += blockDim.x) {
    const int r = i / D, d = i % D, t = t0 + r;
    float val = 0.f;
    if (t < T) {
      switch (g.fmt) {
        case KVQ_FMT_FLOAT:
          val = ld_act(g.pl[P_FULL].p, plane_index(g.pl[P_FULL], b, h, g.H, t, d), g.act);
          break;
        case KVQ_FMT_AFFINE: {
          unsigned c = code_at(plane_ptr<uint8_t>(g, P_CODES, b, h, t), d, bits);
          float s = __half2float(*plane_ptr<__half>(g, P_SCALE, b, h, t, d / G));
          float m = __half2float(*plane_ptr<__half>(g, P_ZERO, b, h, t, d / G));
          val = (float)c * s + m;
          break;
        }
        case KVQ_FMT_SYMMETRIC: {
          unsigned c = code_at(plane_ptr<uint8_t>(g, P_CODES, b, h, t), d, bits);
          float s = __half2float(*plane_ptr<__half>(g, P_SCALE, b, h, t, d / G));
          val = (float)((int)c - (1 << (bits - 1))) * s;
          break;
        }
        case KVQ_FMT_KIVI:
          if (t < tq) {
            unsigned c = code_at(plane_ptr<uint8_t>(g, P_CODES, b, h, t), d, bits);
            float s, m;
            if (which == 0) {
              s = __half2float(*plane_ptr<__half>(g, P_SCALE, b, h, t / G, d));
              m = __half2float(*plane_ptr<__half>(g, P_ZERO, b, h, t / G, d));
            } else {
              s = __half2float(*plane_ptr<__half>(g, P_SCALE, b, h, t, d / G));
              m = __half2float(*plane_ptr<__half>(g, P_ZERO, b, h, t, d / G));
            }
            val = (float)c * s + m;
          } else {
            val = ld_act(g.pl[P_FULL].p, plane_index(g.pl[P_FULL], b, h, g.H, t % g.ring, d),
                         g.act);
          }
          break;
        case KVQ_FMT_KVARN:
          if (t < g.S) {
            val = ld_act(g.pl[P_FULL].p, plane_index(g.pl[P_FULL], b, h, g.H, t, d), g.act);
          } else if (t - g.S < nbq) {
            const int q = t - g.S;
            unsigned c = code_at(plane_ptr<uint8_t>(g, P_CODES, b, h, q), d, bits);
            float s = __half2float(*plane_ptr<__half>(g, P_SCALE, b, h, q, d / G));
            float m = __half2float(*plane_ptr<__half>(g, P_ZERO, b, h, q, d / G));
            float rr = __half2float(*plane_ptr<__half>(g, P_ROW, b, h, 0, q));
            float cc = __half2float(*plane_ptr<__half>(g, P_COL, b, h, q / G, d));
            val = rr * cc * ((float)c * s + m);
          } else {
            val = ld_act(g.pl[P_PEND].p,
                         plane_index(g.pl[P_PEND], b, h, g.H, (t - g.S) % G, d), g.act);
          }
          break;
      }
    }
    dst[r * ld + d] = val;
  }
  if (g.fmt == KVQ_FMT_KVARN && !(t0 >= g.S && t0 + n <= g.S + nbq)) {
    // KVarN is attended in the rotated basis (the coded rows are stored
    // rotated): rotate the full-precision rows (sinks, staged) forward
    __syncthreads();
    for (int hs = 1; hs < D; hs <<= 1) {
      for (int p = threadIdx.x; p < n * D / 2; p += blockDim.x) {
        const int r = p / (D / 2), k = p % (D / 2), t = t0 + r;
        if (t >= T || (t >= g.S && t - g.S < nbq)) continue;
        const int j = (k / hs) * 2 * hs + (k % hs);
        float a = dst[r * ld + j], c = dst[r * ld + j + hs];
        dst[r * ld + j] = a + c;
        dst[r * ld + j + hs] = a - c;
      }
      __syncthreads();
    }
    for (int i = threadIdx.x; i < n * D; i += blockDim.x) {
      const int r = i / D, t = t0 + r;
      if (t < T && !(t >= g.S && t - g.S < nbq)) dst[r * ld + i % D] *= inv_sqrt_d;
    }
  }
}

// Normalised Hadamard transform of `rows` rows of D values at x [rows][ld]
// (the whole CTA; H / sqrt(D) is its own inverse).
__device__ void rotate_rows(float* x, int rows, int D, int ld, float inv_sqrt_d) {
  __syncthreads();
  for (int hs = 1; hs < D; hs <<= 1) {
    for (int p = threadIdx.x; p < rows * D / 2; p += blockDim.x) {
      const int r = p / (D / 2), k = p % (D / 2);
      const int j = (k / hs) * 2 * hs + (k % hs);
      const float a = x[r * ld + j], c = x[r * ld + j + hs];
      x[r * ld + j] = a + c;
      x[r * ld + j + hs] = a - c;
    }
    __syncthreads();
  }
  for (int i = threadIdx.x; i < rows * D; i += blockDim.x) x[(i / D) * ld + i % D] *= inv_sqrt_d;
  __syncthreads();
}

// One CTA: `rows` = g heads x nq queries of one (b, kv head), over the tokens
// [ts, te).  Shared memory holds the K/V tiles, q, scores and accumulators.
// decode: writes (m, l, o) partials to the workspace, else the output.
__global__ void __launch_bounds__(kThreads)
attend_generic_kernel(Geom g, const void* q, int L, float scale, void* out,
                      int nq, int splits, int decode, float inv_sqrt_d) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ float sm[];
  const int T = cache_tokens(g);
  const int D = g.D, grp = g.Hq / g.H;
  const int rows = grp * nq;
  const int ldk = D + 1;
  float* Kt = sm;                       // [kTile][D+1]
  float* Vt = Kt + kTile * ldk;         // [kTile][D]
  float* qs = Vt + kTile * D;           // [rows][D]
  float* acc = qs + rows * D;           // [rows][D]
  float* sc = acc + rows * D;           // [rows][kTile]
  float* mrow = sc + rows * kTile;      // [rows]
  float* lrow = mrow + rows;
  float* arow = lrow + rows;

  const int qtile = blockIdx.x / splits, split = blockIdx.x % splits;
  const int hkv = blockIdx.y, b = blockIdx.z;
  const int q0 = qtile * nq;            // first query of this CTA
  const int nql = min(nq, L - q0);
  const int pos_first = T - L + q0;     // absolute position of query q0
  const int pos_last = pos_first + nql - 1;
  // tokens of this split
  int ts = 0, te = pos_last + 1;
  if (decode) split_range(T, splits, split, kTile, &ts, &te);
  for (int i = threadIdx.x; i < rows * D; i += blockDim.x) {
    const int r = i / D, d = i % D;
    const int hl = r / nq, qi = r % nq;
    const int hq = hkv * grp + hl;
    float v = 0.f;
    if (qi < nql) v = ld_act(q, (((int64_t)b * g.Hq + hq) * L + q0 + qi) * D + d, g.act);
    qs[i] = v;
    acc[i] = 0.f;
  }
  for (int r = threadIdx.x; r < rows; r += blockDim.x) {
    mrow[r] = -INFINITY;
    lrow[r] = 0.f;
  }
  __syncthreads();
  const bool kvarn = g.fmt == KVQ_FMT_KVARN;
  if (kvarn) rotate_rows(qs, rows, D, D, inv_sqrt_d);     // queries into the rotated basis
  for (int t0 = ts; t0 < te; t0 += kTile) {
    const int n = min(kTile, te - t0);
    dequant_tile(g, 0, b, hkv, t0, n, T, Kt, ldk, inv_sqrt_d);
    dequant_tile(g, 1, b, hkv, t0, n, T, Vt, D, inv_sqrt_d);
    __syncthreads();
    for (int i = threadIdx.x; i < rows * kTile; i += blockDim.x) {
      const int r = i / kTile, j = i % kTile;
      const int qi = r % nq;
      const int t = t0 + j;
      float s = -INFINITY;
      if (j < n && qi < nql && t <= pos_first + qi) {
        const float* qr = qs + r * D;
        const float* kr = Kt + j * ldk;
        float a = 0.f;
        for (int d = 0; d < D; ++d) a += qr[d] * kr[d];
        s = a * scale;
      }
      sc[i] = s;
    }
    __syncthreads();
    for (int r = threadIdx.x; r < rows; r += blockDim.x) {
      float mx = -INFINITY;
      for (int j = 0; j < kTile; ++j) mx = fmaxf(mx, sc[r * kTile + j]);
      const float mo = mrow[r];
      const float mn = fmaxf(mo, mx);
      float alpha = 1.f, sum = 0.f;
      if (mn == -INFINITY) {
        for (int j = 0; j < kTile; ++j) sc[r * kTile + j] = 0.f;
      } else {
        alpha = expf(mo - mn);
        for (int j = 0; j < kTile; ++j) {
          const float p = expf(sc[r * kTile + j] - mn);
          sc[r * kTile + j] = p;
          sum += p;
        }
        mrow[r] = mn;
      }
      lrow[r] = lrow[r] * alpha + sum;
      arow[r] = alpha;
    }
    __syncthreads();
    for (int i = threadIdx.x; i < rows * D; i += blockDim.x) {
      const int r = i / D, d = i % D;
      float a = acc[i] * arow[r];
      const float* p = sc + r * kTile;
      for (int j = 0; j < n; ++j) a += p[j] * Vt[j * D + d];
      acc[i] = a;
    }
    __syncthreads();
  }
  if (kvarn) rotate_rows(acc, rows, D, D, inv_sqrt_d);    // output back to the original basis
  if (decode) {
    for (int i = threadIdx.x; i < rows * (D + kWsStride); i += blockDim.x) {
      const int r = i / (D + kWsStride), c = i % (D + kWsStride);
      const int hq = hkv * grp + r;          // nq == 1 in decode
      float* w = ws_row(g, b, hq) + (int64_t)split * (D + kWsStride);
      w[c] = c == 0 ? mrow[r] : c == 1 ? lrow[r] : acc[r * D + c - 2];
    }
  } else {
    for (int i = threadIdx.x; i < rows * D; i += blockDim.x) {
      const int r = i / D, d = i % D;
      const int hl = r / nq, qi = r % nq;
      if (qi >= nql) continue;
      const int hq = hkv * grp + hl;
      const float l = lrow[r];
      st_act(out, (((int64_t)b * g.Hq + hq) * L + q0 + qi) * D + d, acc[i] / l, g.act);
    }
  }
}

// Merge the split partials of one (b, q head): o = sum_s e^(m_s - M) o_s /
// sum_s e^(m_s - M) l_s.
__global__ void combine_kernel(Geom g, int splits, void* out) {
  pdl_wait();
  pdl_trigger();
  const int hq = blockIdx.x, b = blockIdx.y;
  const int D = g.D;
  const float* w = ws_row(g, b, hq);
  float M = -INFINITY;
  for (int s = 0; s < splits; ++s) M = fmaxf(M, w[s * (D + kWsStride)]);
  float Lsum = 0.f;
  for (int s = 0; s < splits; ++s) {
    const float m = w[s * (D + kWsStride)];
    if (m != -INFINITY) Lsum += expf(m - M) * w[s * (D + kWsStride) + 1];
  }
  for (int d = threadIdx.x; d < D; d += blockDim.x) {
    float o = 0.f;
    for (int s = 0; s < splits; ++s) {
      const float m = w[s * (D + kWsStride)];
      if (m != -INFINITY) o += expf(m - M) * w[s * (D + kWsStride) + 2 + d];
    }
    st_act(out, ((int64_t)b * g.Hq + hq) * D + d, o / Lsum, g.act);
  }
}

}  // namespace

int decode_splits(const Geom& g) {
  const int bh = g.B * g.H;
  int s = (2 * num_sms() + bh - 1) / bh;
  if (s > kMaxSplits) s = kMaxSplits;
  return s < 1 ? 1 : s;
}

cudaError_t launch_attend(const Geom& g, const void* q, int L, float scale, void* out,
                          bool decode, cudaStream_t s) {
  if (!decode && prefill_tc_supported(g)) {
    int* err = device_error_word();
    if (!err) return cudaErrorInvalidDevice;
    return launch_prefill_tc(g, q, L, scale, out, err, s);
  }
  if (!decode && prefill_mma_supported(g)) return launch_prefill_mma(g, q, L, scale, out, s);
  if (decode && decode_mma_supported(g)) {
    int* err = device_error_word();
    if (!err) return cudaErrorInvalidDevice;
    return launch_decode_mma(g, q, scale, err, out, s);
  }
  const int grp = g.Hq / g.H;
  const float inv_sqrt_d = (float)(1.0 / sqrt((double)g.D));
  int nq, splits;
  if (decode) {
    nq = 1;
    splits = g.splits;
  } else {
    int rows = 8192 / g.D;
    if (rows > 128) rows = 128;
    nq = rows / grp;
    if (nq < 1) nq = 1;
    splits = 1;
  }
  const int rows = grp * nq;
  const size_t sm = (size_t)(kTile * (g.D + 1) + kTile * g.D + 2 * rows * g.D +
                             rows * kTile + 3 * rows) * sizeof(float);
  cudaError_t e = cudaFuncSetAttribute(attend_generic_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
  if (e != cudaSuccess) return e;
  const int nqt = (L + nq - 1) / nq;
  dim3 grid(nqt * splits, g.H, g.B);
  launch_pdl(attend_generic_kernel, dim3(grid), dim3(kThreads), sm, s, g, q, L, scale, out, nq, splits,
                                                   decode ? 1 : 0, inv_sqrt_d);
  e = cudaGetLastError();
  if (e != cudaSuccess || !decode) return e;
  launch_pdl(combine_kernel, dim3(dim3(g.Hq, g.B)), dim3(64), 0, s, g, splits, out);
  return cudaGetLastError();
}

}  // namespace kvq
