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
// sum_s e^(m_s - M) l_s over slots 0 .. splits-1, and slot `extra` if >= 0.
__global__ void combine_kernel(Geom g, int splits, int extra, void* out) {
  pdl_wait();
  pdl_trigger();
  const int hq = blockIdx.x, b = blockIdx.y;
  const int D = g.D;
  const float* w = ws_row(g, b, hq);
  const int n = splits + (extra >= 0 ? 1 : 0);
  auto row = [&](int i) { return w + (int64_t)(i < splits ? i : extra) * (D + kWsStride); };
  float M = -INFINITY;
  for (int i = 0; i < n; ++i) M = fmaxf(M, row(i)[0]);
  float Lsum = 0.f;
  for (int i = 0; i < n; ++i) {
    const float m = row(i)[0];
    if (m != -INFINITY) Lsum += expf(m - M) * row(i)[1];
  }
  for (int d = threadIdx.x; d < D; d += blockDim.x) {
    float o = 0.f;
    for (int i = 0; i < n; ++i) {
      const float m = row(i)[0];
      if (m != -INFINITY) o += expf(m - M) * row(i)[2 + d];
    }
    st_act(out, ((int64_t)b * g.Hq + hq) * D + d, o / Lsum, g.act);
  }
}

// ---------------------------------------------------------------------------
// KVarN decode attention in the rotated basis (Section 3.1: coded tokens are
// stored as r_t c_j (s code + m) after the normalised Hadamard rotation).
// One CTA = (split, kv head, sequence), 8 warps, each warp a contiguous part
// of the split; lane l holds channels [NS l, NS l + NS), NS = D / 32.  The
// queries are rotated once (in registers); a coded token's score is
//   r_t (s_t sum_j q'_j code_j + m_t sum_j q'_j),  q' = q_rot c_block,
// refolded when the token block changes (a lane's channels lie in one group);
// sinks and staged tokens are rotated forward in registers.  The values
// accumulate in the rotated basis; the split's output is rotated back before
// its (m, l, o) partial goes to the workspace, and the last split CTA of a
// (sequence, kv head) to finish merges the partials into the output.
// ---------------------------------------------------------------------------
template <int D>
__device__ __forceinline__ void fwht_contig(float (&x)[D / 32], int lane, float inv_sqrt_d) {
  constexpr int NS = D / 32;
#pragma unroll
  for (int h = 1; h < NS; h <<= 1)
#pragma unroll
    for (int i = 0; i < NS; ++i)
      if (!(i & h)) {
        const float a = x[i], c = x[i + h];
        x[i] = a + c;
        x[i + h] = a - c;
      }
#pragma unroll
  for (int lh = 1; lh < 32; lh <<= 1)
#pragma unroll
    for (int i = 0; i < NS; ++i) {
      const float y = __shfl_xor_sync(0xffffffffu, x[i], lh);
      x[i] = (lane & lh) ? y - x[i] : x[i] + y;
    }
#pragma unroll
  for (int i = 0; i < NS; ++i) x[i] *= inv_sqrt_d;
}

// NS codes of `bits` bits of this lane's channels from a packed row
__device__ __forceinline__ uint32_t lane_codes(const uint8_t* row, int lane, int ns, int bits) {
  const int bit = ns * bits * lane;
  return __ldg(reinterpret_cast<const uint32_t*>(row) + (bit >> 5)) >> (bit & 31);
}

template <int D, int GM>
__global__ void __launch_bounds__(256)
attend_kvarn_decode_kernel(Geom g, const __nv_bfloat16* __restrict__ q, float scale,
                           float inv_sqrt_d, int full_only, void* out) {
  pdl_wait();
  pdl_trigger();
  constexpr int NS = D / 32;
  extern __shared__ float ksm[];                 // [8 warps][GM][D + 2]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int split = blockIdx.x, hkv = blockIdx.y, b = blockIdx.z;
  const int grp = g.Hq / g.H, G = g.G, S = g.S;
  const int T = cache_tokens(g);
  const int nbq = kvarn_nblocks(T, S, G) * G;
  // full_only: the splits share the full-precision tokens alone (sinks, then
  // staged), indexed f = 0 .. T - nbq - 1 and mapped to token f or f + nbq
  int ts, te;
  if (full_only) split_range(T - nbq, g.splits, split, 1, &ts, &te);
  else split_range(T, g.splits, split, G, &ts, &te);
  const float c2 = scale * 1.4426950408889634f;   // scores in log2 units
  // rotated queries, pre-scaled
  float qr[GM][NS];
#pragma unroll
  for (int h = 0; h < GM; ++h) {
    float x[NS];
    const bool live = h < grp;
    const __nv_bfloat16* src = q + ((int64_t)b * g.Hq + hkv * grp + (live ? h : 0)) * D + NS * lane;
#pragma unroll
    for (int i = 0; i < NS; ++i) x[i] = live ? __bfloat162float(src[i]) : 0.f;
    fwht_contig<D>(x, lane, inv_sqrt_d);
#pragma unroll
    for (int i = 0; i < NS; ++i) qr[h][i] = x[i] * c2;
  }
  float m[GM], l[GM], o[GM][NS];
#pragma unroll
  for (int h = 0; h < GM; ++h) {
    m[h] = -INFINITY;
    l[h] = 0.f;
#pragma unroll
    for (int i = 0; i < NS; ++i) o[h][i] = 0.f;
  }
  const int per = (te - ts + 7) / 8;
  const int w0 = ts + warp * per, w1 = min(te, w0 + per);
  const int kb = g.kb, vb = g.vb;
  const unsigned kmask = (1u << kb) - 1, vmask = (1u << vb) - 1;
  const int grpc = NS * lane / G;                   // this lane's channel group
  float qp[GM][NS], qs[GM];                         // q' = q_rot c_block and its lane sum
  float cv[NS];                                     // value column scales of the block
  int cur_blk = -1;
  for (int f = w0; f < w1; ++f) {
    const int t = full_only && f >= S ? f + nbq : f;
    float kv[NS], vv[NS];
    const bool coded = t >= S && t - S < nbq;
    float dot[GM];
    if (coded) {
      const int qi = t - S, blk = qi / G;
      if (blk != cur_blk) {                         // refold the block's column scales
        cur_blk = blk;
        const __half* ck = plane_ptr<__half>(g, KVQ_PLANE_K_COL, b, hkv, blk, NS * lane);
        const __half* cvp = plane_ptr<__half>(g, KVQ_PLANE_V_COL, b, hkv, blk, NS * lane);
#pragma unroll
        for (int i = 0; i < NS; ++i) {
          const float c = __half2float(ck[i]);
          cv[i] = __half2float(cvp[i]);
#pragma unroll
          for (int h = 0; h < GM; ++h) qp[h][i] = qr[h][i] * c;
        }
#pragma unroll
        for (int h = 0; h < GM; ++h) {
          float a = 0.f;
#pragma unroll
          for (int i = 0; i < NS; ++i) a += qp[h][i];
          qs[h] = a;
        }
      }
      const uint32_t wk = lane_codes(plane_ptr<uint8_t>(g, KVQ_PLANE_K_CODES, b, hkv, qi), lane, NS, kb);
      const uint32_t wv = lane_codes(plane_ptr<uint8_t>(g, KVQ_PLANE_V_CODES, b, hkv, qi), lane, NS, vb);
      const float ks = __half2float(*plane_ptr<__half>(g, KVQ_PLANE_K_SCALE, b, hkv, qi, grpc));
      const float kz = __half2float(*plane_ptr<__half>(g, KVQ_PLANE_K_ZERO, b, hkv, qi, grpc));
      const float kr = __half2float(*plane_ptr<__half>(g, KVQ_PLANE_K_ROW, b, hkv, 0, qi));
      const float vs = __half2float(*plane_ptr<__half>(g, KVQ_PLANE_V_SCALE, b, hkv, qi, grpc));
      const float vz = __half2float(*plane_ptr<__half>(g, KVQ_PLANE_V_ZERO, b, hkv, qi, grpc));
      const float vr = __half2float(*plane_ptr<__half>(g, KVQ_PLANE_V_ROW, b, hkv, 0, qi));
#pragma unroll
      for (int h = 0; h < GM; ++h) {
        float a = 0.f;
#pragma unroll
        for (int i = 0; i < NS; ++i) a += qp[h][i] * (float)((wk >> (i * kb)) & kmask);
        dot[h] = kr * (ks * a + kz * qs[h]);
      }
#pragma unroll
      for (int i = 0; i < NS; ++i) vv[i] = vr * cv[i] * ((float)((wv >> (i * vb)) & vmask) * vs + vz);
    } else {                                        // sink or staged: rotate forward
      const __nv_bfloat16* kp = t < S
          ? plane_ptr<__nv_bfloat16>(g, KVQ_PLANE_K_FULL, b, hkv, t, NS * lane)
          : plane_ptr<__nv_bfloat16>(g, KVQ_PLANE_K_PEND, b, hkv, (t - S) % G, NS * lane);
      const __nv_bfloat16* vp = t < S
          ? plane_ptr<__nv_bfloat16>(g, KVQ_PLANE_V_FULL, b, hkv, t, NS * lane)
          : plane_ptr<__nv_bfloat16>(g, KVQ_PLANE_V_PEND, b, hkv, (t - S) % G, NS * lane);
#pragma unroll
      for (int i = 0; i < NS; ++i) {
        kv[i] = __bfloat162float(kp[i]);
        vv[i] = __bfloat162float(vp[i]);
      }
      fwht_contig<D>(kv, lane, inv_sqrt_d);
      fwht_contig<D>(vv, lane, inv_sqrt_d);
#pragma unroll
      for (int h = 0; h < GM; ++h) {
        float a = 0.f;
#pragma unroll
        for (int i = 0; i < NS; ++i) a += qr[h][i] * kv[i];
        dot[h] = a;
      }
    }
#pragma unroll
    for (int h = 0; h < GM; ++h) {
      float sc = dot[h];
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) sc += __shfl_xor_sync(0xffffffffu, sc, off);
      const float mn = fmaxf(m[h], sc);
      const float alpha = exp2f(m[h] - mn);         // m = -inf at first: alpha = 0
      const float p = exp2f(sc - mn);
      m[h] = mn;
      l[h] = l[h] * alpha + p;
#pragma unroll
      for (int i = 0; i < NS; ++i) o[h][i] = o[h][i] * alpha + p * vv[i];
    }
  }
  // ---- merge the warps, rotate back, write the split's partial ----
  float* red = ksm;                                  // [8][GM][D + 2]
#pragma unroll
  for (int h = 0; h < GM; ++h) {
    float* rw = red + (warp * GM + h) * (D + 2);
    if (lane == 0) {
      rw[0] = m[h];
      rw[1] = l[h];
    }
#pragma unroll
    for (int i = 0; i < NS; ++i) rw[2 + NS * lane + i] = o[h][i];
  }
  __syncthreads();
  for (int h = warp; h < grp; h += 8) {
    float M = -INFINITY;
    for (int w = 0; w < 8; ++w) M = fmaxf(M, red[(w * GM + h) * (D + 2)]);
    float L = 0.f, x[NS];
#pragma unroll
    for (int i = 0; i < NS; ++i) x[i] = 0.f;
    for (int w = 0; w < 8; ++w) {
      const float* rw = red + (w * GM + h) * (D + 2);
      if (rw[0] == -INFINITY) continue;
      const float f = exp2f(rw[0] - M);
      L += f * rw[1];
#pragma unroll
      for (int i = 0; i < NS; ++i) x[i] += f * rw[2 + NS * lane + i];
    }
    fwht_contig<D>(x, lane, inv_sqrt_d);
    float* wsr = ws_row(g, b, hkv * grp + h) + (int64_t)split * (D + kWsStride);
    if (lane == 0) {
      wsr[0] = M == -INFINITY ? -INFINITY : M * 0.6931471805599453f;   // natural-log units
      wsr[1] = L;
    }
#pragma unroll
    for (int i = 0; i < NS; ++i) wsr[2 + NS * lane + i] = x[i];
  }
  // ---- the last split CTA of this (sequence, kv head) merges the splits
  // and, with full_only, the coded tokens' partial (slot kMaxSplits - 1,
  // written by the streaming kernel that ran before this one) ----
  __shared__ int last_cta;
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    last_cta = atomicAdd(&g.counters[b * g.H + hkv], 1u) == (unsigned)g.splits - 1;
  }
  __syncthreads();
  if (!last_cta) return;
  __threadfence();
  const int n = g.splits + (full_only ? 1 : 0);
  for (int h = warp; h < grp; h += 8) {
    const float* w = ws_row(g, b, hkv * grp + h);
    auto row = [&](int i) { return w + (int64_t)(i < g.splits ? i : kMaxSplits - 1) * (D + kWsStride); };
    float M = -INFINITY;
    for (int i = lane; i < n; i += 32) M = fmaxf(M, __ldcg(row(i)));
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
    float L = 0.f, acc[NS];
#pragma unroll
    for (int i = 0; i < NS; ++i) acc[i] = 0.f;
    for (int i = 0; i < n; ++i) {
      const float mi = __ldcg(row(i));
      if (mi == -INFINITY) continue;
      const float f = expf(mi - M);
      L += f * __ldcg(row(i) + 1);
#pragma unroll
      for (int k = 0; k < NS; ++k) acc[k] += f * __ldcg(row(i) + 2 + lane + 32 * k);
    }
#pragma unroll
    for (int k = 0; k < NS; ++k)
      st_act(out, ((int64_t)b * g.Hq + hkv * grp + h) * D + lane + 32 * k, acc[k] / L, g.act);
  }
  if (threadIdx.x == 0) g.counters[b * g.H + hkv] = 0;   // ready for the next call
}

template <int D>
cudaError_t launch_kvarn_d(const Geom& g, const void* q, float scale, int full_only, void* out,
                           cudaStream_t s) {
  const int grp = g.Hq / g.H;
  const float inv_sqrt_d = (float)(1.0 / sqrt((double)D));
  dim3 grid(g.splits, g.H, g.B);
  auto run = [&](auto kern, int gm) {
    const size_t sm = (size_t)8 * gm * (D + 2) * sizeof(float);
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
    if (e != cudaSuccess) return e;
    launch_pdl(kern, dim3(grid), dim3(256), sm, s, g, reinterpret_cast<const __nv_bfloat16*>(q),
               scale, inv_sqrt_d, full_only, out);
    return cudaGetLastError();
  };
  if (grp <= 2) return run(attend_kvarn_decode_kernel<D, 2>, 2);
  if (grp <= 4) return run(attend_kvarn_decode_kernel<D, 4>, 4);
  return run(attend_kvarn_decode_kernel<D, 8>, 8);
}

bool kvarn_decode_supported(const Geom& g) {
  return g.fmt == KVQ_FMT_KVARN && g.act == KVQ_BF16 && (g.D == 64 || g.D == 128 || g.D == 256) &&
         g.Hq / g.H <= 8 && (g.kb == 2 || g.kb == 4) && (g.vb == 2 || g.vb == 4) &&
         g.G >= g.D / 32 && g.G % (g.D / 32) == 0;
}

}  // namespace

int decode_splits(const Geom& g) {
  // the split kernels fit two CTAs per SM: round down so that every split of
  // every (sequence, kv head) runs in the first wave
  const int bh = g.B * g.H;
  int s = 2 * num_sms() / bh;
  if (s > kMaxSplits - 1) s = kMaxSplits - 1;     // the last slot is reserved (KVarN)
  return s < 1 ? 1 : s;
}

cudaError_t launch_attend(const Geom& g, const void* q, int L, float scale, void* out,
                          bool decode, int t_hint, cudaStream_t s) {
  if (!decode && prefill_m256_supported(g)) {
    int* err = device_error_word();
    if (!err) return cudaErrorInvalidDevice;
    return launch_prefill_m256(g, q, L, scale, out, err, s);
  }
  if (!decode && prefill_mma_supported(g)) return launch_prefill_mma(g, q, L, scale, out, s);
  // the streaming decode pays off once every CTA streams a few stages; short
  // caches keep the split kernel (both read T on the device and are exact
  // for any T, so a captured graph stays correct as the cache grows)
  const int64_t blocks = (int64_t)g.B * g.H * ((t_hint + 31) / 32);
  if (decode && decode_stream_supported(g) &&
      (!decode_mma_supported(g) || blocks >= 16 * (int64_t)decode_stream_ctas(g))) {
    int* err = device_error_word();
    if (!err) return cudaErrorInvalidDevice;
    return launch_decode_stream(g, q, scale, err, out, s);
  }
  if (decode && decode_mma_supported(g)) {
    int* err = device_error_word();
    if (!err) return cudaErrorInvalidDevice;
    return launch_decode_mma(g, q, scale, err, out, s);
  }
  if (decode && kvarn_decode_supported(g)) {
    // long caches: the coded tokens on tensor cores (one partial per head in
    // the reserved slot), the sinks and staged tokens in the split kernel
    const int64_t coded = (int64_t)g.B * g.H * (kvarn_nblocks(t_hint, g.S, g.G) * g.G / 32);
    const bool streamed = decode_stream_kvarn_supported(g) &&
                          coded >= 16 * (int64_t)decode_stream_ctas(g);
    if (streamed) {
      int* err = device_error_word();
      if (!err) return cudaErrorInvalidDevice;
      cudaError_t e = launch_decode_stream_kvarn(g, q, scale, err, s);
      if (e != cudaSuccess) return e;
    }
    // the split kernel's last CTA per (sequence, kv head) merges everything
    return g.D == 64 ? launch_kvarn_d<64>(g, q, scale, streamed, out, s)
         : g.D == 128 ? launch_kvarn_d<128>(g, q, scale, streamed, out, s)
                      : launch_kvarn_d<256>(g, q, scale, streamed, out, s);
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
  launch_pdl(combine_kernel, dim3(dim3(g.Hq, g.B)), dim3(64), 0, s, g, splits, -1, out);
  return cudaGetLastError();
}

}  // namespace kvq
