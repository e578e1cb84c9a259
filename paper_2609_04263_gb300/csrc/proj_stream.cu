// Few-row (decode) LoRA Q/K/V projection as one weight stream (Section 3,
// Eq. 1 and the LoRA update): Y_p = X W_p^T + (alpha/r) (X A_p^T) B_p^T, then
// RoPE on queries and keys, for M = B * L <= 16 rows of X in bf16.
//
// A decode step reads every weight once and computes almost nothing, so the
// kernel is a copy at HBM speed with a few MMAs riding on it:
//   * one CTA per SM; the RoPE pair-tiles (8 channels of one head and their
//     partners D/2 further, 16 weight rows) are cut into contiguous ranges,
//     one per CTA;
//   * each tile streams through a ring of shared stages as two stages of 8
//     whole weight rows, each one contiguous cp.async.bulk of 16 d_in bytes
//     (with 18 row copies per stage the refilling warp held the other warps
//     at the tile-end barrier), and
//     the tile's 16 rows of B_p ride with its second stage; there is no
//     producer warp: the last warp to finish with a stage (a shared counter)
//     refills it at once with the stage ns further on;
//   * the 16 warps hold the rows of X in registers, each warp the same
//     32-channel chunks of every stage, so no shared memory goes to X;
//     X is the MMA's A operand (tokens as rows), the weight rows are B
//     operands (n = 8 rows), and within a 32-channel chunk the k index is
//     permuted so that every operand is one 16-byte load;
//   * before its pair-tiles, each CTA computes U_p = X A_p^T for the
//     projections its range touches, streaming A_p through the same ring as
//     16-row tiles, and keeps U in shared memory for the epilogues;
//   * at a tile's end the warps' partial tiles are summed through shared
//     memory; (alpha/r) U B^T, RoPE and the head-major bf16 store follow.
// Every mbarrier wait is bounded; a timeout sets the library's error word.
#include "proj_decode.cuh"
#include "decode_attn.cuh"

namespace kvq {
namespace {

using pdec::ProjArgs;
using pdec::rope_cos_sin;

constexpr int kCW = 16;                    // warps (all consume; the last one out refills)
constexpr int kPThreads = kCW * 32;
constexpr int kMaxK = 4096;                // input channels (X chunks held per warp: kMaxK / 512)
constexpr int kXC = kMaxK / (32 * kCW);    // 32-channel chunks of X per warp
constexpr int kMaxNS = 8;                  // ring stages
constexpr int kSmemMax = 227 * 1024;

struct PSLayout {
  int ns, stage, wb, rmax;
  int red, fin, us, ring, total;
};

PSLayout ps_layout(int M16, int K, int rmax) {
  PSLayout L;
  L.rmax = rmax;
  L.red = kMaxNS * 8 + kMaxNS * 4 + 16;                   // mbarriers, counters, flags
  L.fin = L.red + kCW * 2 * 32 * 4 * 4;                    // [warps][2][32 lanes][4]
  L.us = L.fin + 16 * 16 * 4;                              // [16 m][16 n]
  L.ring = (L.us + 3 * M16 * (rmax > 0 ? rmax : 1) * 4 + 127) & ~127;   // U [3][M16][rmax]
  L.wb = 16 * K;                                           // B rows after the 8 weight rows
  L.stage = (L.wb + 32 * rmax + 127) & ~127;
  L.ns = (kSmemMax - L.ring) / L.stage;
  if (L.ns > kMaxNS) L.ns = kMaxNS;
  L.total = L.ring + L.ns * L.stage;
  return L;
}

struct Tile {
  int u;      // 1: 16 rows of A_p (U tile); 0: a RoPE pair-tile of W
  int p;      // projection 0 q, 1 k, 2 v
  int j0;     // U tile: first rank row
  int rows;   // rows copied
  int hh;     // pair-tile: stacked head (queries, then keys, then values)
  int head;   // head within its projection
  int c0;     // pair-tile: first channel (its partners are c0 + D/2 ...)
};

__device__ __forceinline__ int proj_of(const ProjArgs& a, int hh) {
  return hh < a.Hq ? 0 : hh < a.Hq + a.Hkv ? 1 : 2;
}

// Tile ti of a CTA whose pair-tiles are [t0, t1): first the U tiles of the
// projections plo..phi (those with rank > 0), then the pair-tiles.
__device__ __forceinline__ Tile tile_at(const ProjArgs& a, int ti, int plo, int phi, int nut,
                                        int t0, int tph) {
  Tile t;
  t.u = 0;
  t.j0 = 0;
  if (ti < nut) {
    int i = ti;
    for (int q = plo; q <= phi; ++q) {
      const int n = (a.r[q] + 15) >> 4;
      if (i < n) {
        t.u = 1;
        t.p = q;
        t.j0 = 16 * i;
        t.rows = min(16, a.r[q] - t.j0);
        t.hh = t.head = t.c0 = 0;
        return t;
      }
      i -= n;
    }
  }
  const int T = t0 + ti - nut;
  t.hh = T / tph;
  t.c0 = (T - t.hh * tph) * 8;
  t.p = proj_of(a, t.hh);
  t.head = t.p == 0 ? t.hh : t.p == 1 ? t.hh - a.Hq : t.hh - a.Hq - a.Hkv;
  t.rows = 16;
  return t;
}

__device__ __forceinline__ void csync() {
  asm volatile("bar.sync 1, %0;" ::"n"(kCW * 32) : "memory");
}

// Copies of stage s (tile s / 2, rows 8 (s % 2) .. of it) into its ring slot:
// lane 0 copies the 8 contiguous weight rows, lanes 1 and 2 the two 8-row
// blocks of B_p with a pair-tile's second stage.  Called by a whole warp.
__device__ void issue_stage(const ProjArgs& a, const PSLayout& L, int s, int plo, int phi,
                            int nut, int t0, int tph, uint64_t* full, unsigned char* ring,
                            int lane) {
  const int K = a.d_in, D = a.D, half = D / 2;
  const int st = s % L.ns, ti = s >> 1, hf = s & 1;
  const Tile t = tile_at(a, ti, plo, phi, nut, t0, tph);
  const int r = a.r[t.p];
  const int rows = t.u ? max(0, min(8, r - t.j0 - 8 * hf)) : 8;
  const bool bcopy = !t.u && r > 0 && hf == 1;
  unsigned char* sp = ring + (size_t)st * L.stage;
  if (lane == 0) {
    // the slot was last read through the generic proxy; the copies write it
    // through the async proxy
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    dattn::mbar_expect_tx(&full[st], (uint32_t)(rows * K * 2 + (bcopy ? 32 * r : 0)));
    if (rows > 0) {
      const __nv_bfloat16* src =
          t.u ? reinterpret_cast<const __nv_bfloat16*>(a.a[t.p]) + (int64_t)(t.j0 + 8 * hf) * K
              : reinterpret_cast<const __nv_bfloat16*>(a.w) +
                    ((int64_t)t.hh * D + hf * half + t.c0) * K;
      dattn::bulk_g2s(sp, src, (uint32_t)(rows * K * 2), &full[st]);
    }
  }
  __syncwarp();
  if (bcopy && (lane == 1 || lane == 2)) {
    const int j = lane - 1;
    const __nv_bfloat16* Bm = reinterpret_cast<const __nv_bfloat16*>(a.bm[t.p]);
    const int c = j == 0 ? t.c0 : half + t.c0;
    dattn::bulk_g2s(sp + L.wb + j * 16 * r, Bm + ((int64_t)t.head * D + c) * r,
                    (uint32_t)(16 * r), &full[st]);
  }
}

__device__ __forceinline__ uint4 lds128(const unsigned char* p) {
  return *reinterpret_cast<const uint4*>(p);
}

template <int M16>   // rows of X held: 8 (M <= 8) or 16
__global__ void __launch_bounds__(kPThreads, 1)
project_decode_stream_kernel(const ProjArgs a, const PSLayout L, int* err) {
  extern __shared__ __align__(128) unsigned char smem[];
  uint64_t* full = reinterpret_cast<uint64_t*>(smem);
  float* red = reinterpret_cast<float*>(smem + L.red);
  float* fin = reinterpret_cast<float*>(smem + L.fin);
  float* us = reinterpret_cast<float*>(smem + L.us);
  unsigned char* ring = smem + L.ring;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int K = a.d_in, D = a.D, half = D / 2, tph = D / 16;
  const int N = (a.Hq + 2 * a.Hkv) * tph;                  // pair-tiles
  const int P = gridDim.x;                                 // <= N (host)
  const int t0 = (int)((int64_t)blockIdx.x * N / P);
  const int t1 = (int)((int64_t)(blockIdx.x + 1) * N / P);
  const int plo = proj_of(a, t0 / tph), phi = proj_of(a, (t1 - 1) / tph);
  int nut = 0;
  for (int q = plo; q <= phi; ++q) nut += (a.r[q] + 15) >> 4;
  const int ntl = nut + (t1 - t0);
  const int nst = 2 * ntl;                                 // two 8-row stages per tile
  const int ns = L.ns;

  uint32_t* cnt = reinterpret_cast<uint32_t*>(full + kMaxNS);   // warps done per slot
  int* flags = reinterpret_cast<int*>(cnt + kMaxNS);          // [0] bad, [1] stages issued
  if (threadIdx.x == 0) {
    for (int i = 0; i < ns; ++i) {
      dattn::mbar_init(&full[i], 1);
      cnt[i] = 0;
    }
    flags[0] = 0;
    flags[1] = min(ns, nst);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  pdl_wait();
  pdl_trigger();
  if (warp < min(ns, nst)) issue_stage(a, L, warp, plo, phi, nut, t0, tph, full, ring, lane);

  // ---------------------------------------------------------------- consumers
  // a warp done with stage s counts itself out of the slot; the last one
  // refills the slot with stage s + ns
  auto release = [&](int s) {
    __syncwarp();
    uint32_t old = 0;
    if (lane == 0) {
      __threadfence_block();
      old = atomicAdd(&cnt[s % ns], 1u);
    }
    old = __shfl_sync(0xffffffffu, old, 0);
    if (old == kCW - 1) {
      __threadfence_block();
      if (lane == 0) {
        cnt[s % ns] = 0;
        if (s + ns < nst) atomicMax(&flags[1], s + ns + 1);
      }
      if (s + ns < nst) issue_stage(a, L, s + ns, plo, phi, nut, t0, tph, full, ring, lane);
    }
  };
  const int gid = lane >> 2, tid = lane & 3, tc = threadIdx.x;
  const int M = a.B * a.L;
  const __nv_bfloat16* x = reinterpret_cast<const __nv_bfloat16*>(a.x);
  // this warp's chunks of X: chunk warp + 16 h, channels 8 tid .. 8 tid + 7
  const int nch = K / 32;
  uint4 xa[kXC], xb[kXC];
#pragma unroll
  for (int h = 0; h < kXC; ++h) {
    const int k = (warp + 16 * h) * 32 + 8 * tid;
    xa[h] = xb[h] = make_uint4(0, 0, 0, 0);
    if (k < K && gid < M) xa[h] = __ldg(reinterpret_cast<const uint4*>(x + (int64_t)gid * K + k));
    if (M16 == 16 && k < K && gid + 8 < M)
      xb[h] = __ldg(reinterpret_cast<const uint4*>(x + (int64_t)(gid + 8) * K + k));
  }
  float acc[2][4];
#pragma unroll
  for (int n = 0; n < 2; ++n) acc[n][0] = acc[n][1] = acc[n][2] = acc[n][3] = 0.f;
  bool bad = false;

  for (int ti = 0; ti < ntl; ++ti) {
    const Tile t = tile_at(a, ti, plo, phi, nut, t0, tph);
    int st = 0;
#pragma unroll
    for (int hf = 0; hf < 2; ++hf) {        // weight rows 0..7, then 8..15
      {
        const int s = 2 * ti + hf;
        st = s % ns;
        if (!bad) {
          bool ok = true;
          if (lane == 0) ok = dattn::mbar_wait(&full[st], (s / ns) & 1);
          if (!__shfl_sync(0xffffffffu, ok, 0)) {
            if (lane == 0) atomicOr(err, 1);
            bad = true;
          }
        }
        if (!bad) {
          // rows are 2 K bytes apart: a quarter-warp's two rows share banks
          // (two-way), which the idle consumers absorb
          const unsigned char* sp = ring + (size_t)st * L.stage + gid * (2 * K) + 16 * tid;
#pragma unroll
          for (int h = 0; h < kXC; ++h) {
            const int j = warp + 16 * h;
            if (j < nch) {
              const uint4 w = lds128(sp + j * 64);
              const uint4 p = xa[h], q = xb[h];
              pdec::mma16816_p(acc[hf], p.x, q.x, p.y, q.y, w.x, w.y);
              pdec::mma16816_p(acc[hf], p.z, q.z, p.w, q.w, w.z, w.w);
            }
          }
          if (hf == 0) release(s);
        }
      }
    }
    // ---- tile end: sum the warps' partial tiles
#pragma unroll
    for (int n = 0; n < 2; ++n) {
      *reinterpret_cast<float4*>(red + ((warp * 2 + n) * 32 + lane) * 4) =
          make_float4(acc[n][0], acc[n][1], acc[n][2], acc[n][3]);
      acc[n][0] = acc[n][1] = acc[n][2] = acc[n][3] = 0.f;
    }
    csync();
    if (tc < M16 * 16) {
      // fragment element i of lane ln holds (m, n) = (ln/4 + 8 (i/2), 2 (ln%4) + i%2)
      const int m = tc >> 4, n = tc & 15, nt = n >> 3, col = n & 7;
      const int ln = (m & 7) * 4 + (col >> 1), i = ((m >> 3) << 1) | (col & 1);
      float sum = 0.f;
#pragma unroll
      for (int w = 0; w < kCW; ++w) sum += red[((w * 2 + nt) * 32 + ln) * 4 + i];
      fin[m * 16 + n] = sum;
    }
    csync();
    const int r = a.r[t.p];
    if (t.u) {
      if (tc < M * 16) {
        const int m = tc >> 4, j = tc & 15;
        if (t.j0 + j < r) us[(t.p * M16 + m) * L.rmax + t.j0 + j] = fin[m * 16 + j];
      }
    } else if (tc < M * 8) {
      const int m = tc >> 3, i = tc & 7;
      float y1 = fin[m * 16 + i], y2 = fin[m * 16 + 8 + i];
      if (r > 0) {
        const unsigned char* bs = ring + (size_t)st * L.stage + L.wb;
        const __nv_bfloat16* b1 = reinterpret_cast<const __nv_bfloat16*>(bs) + i * r;
        const __nv_bfloat16* b2 = reinterpret_cast<const __nv_bfloat16*>(bs) + (8 + i) * r;
        const float* u = us + (t.p * M16 + m) * L.rmax;
        for (int j0 = 0; j0 < r; j0 += 8) {
          const uint4 u1 = *reinterpret_cast<const uint4*>(b1 + j0);
          const uint4 u2 = *reinterpret_cast<const uint4*>(b2 + j0);
          const __nv_bfloat16* e1 = reinterpret_cast<const __nv_bfloat16*>(&u1);
          const __nv_bfloat16* e2 = reinterpret_cast<const __nv_bfloat16*>(&u2);
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const float uu = u[j0 + e] * a.alpha_over_r;
            y1 += uu * __bfloat162float(e1[e]);
            y2 += uu * __bfloat162float(e2[e]);
          }
        }
      }
      const int b = m / a.L, l = m - b * a.L;
      const int c = t.c0 + i;
      if (t.p < 2 && a.rope_base > 0.f) {
        float cs, sn;
        rope_cos_sin(a.pos0 + pos_of(a.pos_dev, a.pos_stride, b) + l, a.theta_hi[c],
                     a.theta_lo[c], &cs, &sn);
        const float o1 = y1 * cs - y2 * sn, o2 = y2 * cs + y1 * sn;
        y1 = o1;
        y2 = o2;
      }
      const int H = t.p == 0 ? a.Hq : a.Hkv;
      __nv_bfloat16* out = reinterpret_cast<__nv_bfloat16*>(a.out[t.p]);
      const int64_t base = (((int64_t)b * H + t.head) * a.L + l) * D;
      if (!bad) {
        out[base + c] = __float2bfloat16_rn(y1);
        out[base + c + half] = __float2bfloat16_rn(y2);
      }
    }
    // the tile's last stage (its B rows were read above) goes back to the ring
    if (!bad) release(2 * ti + 1);
  }
  // after a timeout, keep the CTA alive until the copies it started have landed
  if (bad && lane == 0) atomicOr(&flags[0], 1);
  csync();
  if (flags[0] && threadIdx.x == 0) {
    const int issued = flags[1];
    for (int i = max(0, issued - ns); i < issued; ++i)
      if (!dattn::mbar_wait(&full[i % ns], (i / ns) & 1)) atomicOr(err, 1);
  }
}

template <int M16>
cudaError_t launch_ps(const ProjArgs& p, const PSLayout& L, int* err, cudaStream_t s) {
  auto kern = project_decode_stream_kernel<M16>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, L.total);
  if (e != cudaSuccess) return e;
  const int N = (p.Hq + 2 * p.Hkv) * (p.D / 16);
  const int P = min(num_sms(), N);
  launch_pdl(kern, dim3(P), dim3(kPThreads), (size_t)L.total, s, p, L, err);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_project_decode_stream(const ProjArgs& p, int* err, cudaStream_t s) {
  const int M = p.B * p.L;
  if (M < 1 || M > 16 || p.d_in % 64 || p.d_in > kMaxK) return cudaErrorNotSupported;
  int rmax = 0;
  for (int i = 0; i < 3; ++i) rmax = max(rmax, p.r[i]);
  if (rmax > 64) return cudaErrorNotSupported;
  const PSLayout L = ps_layout(M <= 8 ? 8 : 16, p.d_in, rmax);
  if (L.ns < 2) return cudaErrorNotSupported;
  return M <= 8 ? launch_ps<8>(p, L, err, s) : launch_ps<16>(p, L, err, s);
}

}  // namespace kvq
