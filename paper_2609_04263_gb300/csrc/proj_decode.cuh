// Device code of the few-row (decode) projection: shared by the standalone
// kernel in project.cu and the fused decode step in decode_step.cu.
#pragma once

#include <math.h>

#include "kvq_internal.cuh"

namespace kvq {
namespace pdec {

struct ProjArgs {
  const void* x;
  const void* w;
  const void* a[3];
  const void* bm[3];
  int r[3];
  void* out[3];
  int B, L, d_in, Hq, Hkv, D, pos0, act;
  const int* pos_dev;   // if set, positions start at pos_of(pos_dev, pos_stride, b) + pos0
  int pos_stride;
  float alpha_over_r, rope_base;
  // RoPE frequencies base^(-2i/D), i < D/2, computed in fp64 on the host and
  // split into hi + lo floats
  float theta_hi[128], theta_lo[128];
};

// cos and sin of pos * theta in fp32 for positions below 2^24: pos * theta_hi
// is formed exactly as p + e (FMA), reduced by 2 pi in three parts (the first
// exact for multiples below 2^15) to |r| <= pi, where the hardware __sincosf
// is accurate to about 2^-21 absolute (far below the bf16 rounding of the
// outputs) without the large-argument path of sincosf.
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
  __sincosf(r, s, c);
}

// ---------------------------------------------------------------------------
// Few rows (M = B * L <= 16, the decode step), bf16: weight streaming on
// mma.sync.  One CTA per RoPE pair-tile: weight rows hD + c0 + i and their
// partners hD + D/2 + c0 + i (i < 8) of one head, plus the rank rows of A_p.
// x is the MMA's A operand (tokens as rows, zero-padded to 16); weight rows
// are B operands (n = 8 rows).  Within each 32-channel chunk the MMA k index
// is permuted so that a thread's operand is one 16-byte load: thread t holds
// channels 8t .. 8t+7, words 2s and 2s+1 feed k-step s.  The 8 warps split
// the channels; partial tiles are summed through shared memory, then the
// rank-r up-projection, RoPE and the head-major store follow.
// ---------------------------------------------------------------------------
constexpr int kDecWarps = 8;
constexpr int kDecMaxNt = 2 + 8;          // 2 weight tiles + up to 64 ranks / 8

__device__ __forceinline__ void mma16816_p(float c[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                           uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// One pair-tile; blockIdx-independent so that a fused kernel can run several
// per CTA.  dsm: at least proj_decode_smem_bytes(M16, NT, d_in) bytes.
template <int M16, int NT>   // M16: x rows held (8 or 16); NT: 2 + rank tiles
__device__ void proj_decode_tile(const ProjArgs& p, int tile, unsigned char* dsm) {
  const int M = p.B * p.L, D = p.D, K = p.d_in;
  const int half = D / 2;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gid = lane >> 2, tid = lane & 3;
  const int tiles_per_head = half / 8;
  const int hh = tile / tiles_per_head;                     // stacked head index
  const int c0 = (tile % tiles_per_head) * 8;
  const int proj = hh < p.Hq ? 0 : hh < p.Hq + p.Hkv ? 1 : 2;
  const int head = proj == 0 ? hh : proj == 1 ? hh - p.Hq : hh - p.Hq - p.Hkv;
  const int r = p.r[proj];
  const int nt_used = 2 + r / 8;                            // r is a multiple of 8
  __nv_bfloat16* xs = reinterpret_cast<__nv_bfloat16*>(dsm);   // [M16][K]
  float* red = reinterpret_cast<float*>(dsm + (size_t)M16 * K * 2);   // [warps][NT][32][4]
  float* fin = red + kDecWarps * NT * 128;                  // [NT][16 m][8 n]
  const __nv_bfloat16* x = reinterpret_cast<const __nv_bfloat16*>(p.x);
  const __nv_bfloat16* W = reinterpret_cast<const __nv_bfloat16*>(p.w);
  const __nv_bfloat16* A = reinterpret_cast<const __nv_bfloat16*>(p.a[proj]);

  // x -> shared memory (rows >= M zero)
  for (int i = threadIdx.x * 8; i < M16 * K; i += blockDim.x * 8) {
    uint4 v = make_uint4(0, 0, 0, 0);
    if (i < M * K) v = __ldg(reinterpret_cast<const uint4*>(x + i));
    *reinterpret_cast<uint4*>(xs + i) = v;
  }
  // B-operand row pointers of this thread (row gid of each n-tile)
  const __nv_bfloat16* brow[NT];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) {
    if (nt == 0) brow[nt] = W + ((int64_t)hh * D + c0 + gid) * K;
    else if (nt == 1) brow[nt] = W + ((int64_t)hh * D + half + c0 + gid) * K;
    else brow[nt] = A + (int64_t)((nt - 2) * 8 + gid) * K;   // valid only for nt < nt_used
  }
  __syncthreads();
  float acc[NT][4];
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) acc[nt][0] = acc[nt][1] = acc[nt][2] = acc[nt][3] = 0.f;
  const int chunks = K / 32;
  const int per = (chunks + kDecWarps - 1) / kDecWarps;
  const int ch0 = warp * per, ch1 = min(chunks, ch0 + per);
  constexpr int U = 4;                                       // chunks in flight per pass
  for (int cb = ch0; cb < ch1; cb += U) {
    uint4 bw[U][NT];
#pragma unroll
    for (int u = 0; u < U; ++u)
#pragma unroll
      for (int nt = 0; nt < NT; ++nt)
        if (cb + u < ch1 && nt < nt_used)
          bw[u][nt] = __ldg(reinterpret_cast<const uint4*>(brow[nt] + (cb + u) * 32 + 8 * tid));
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (cb + u >= ch1) break;
      const int k = (cb + u) * 32 + 8 * tid;
      const uint4 xa = *reinterpret_cast<const uint4*>(xs + gid * K + k);
      uint4 xb = make_uint4(0, 0, 0, 0);
      if (M16 == 16) xb = *reinterpret_cast<const uint4*>(xs + (gid + 8) * K + k);
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        if (nt < nt_used) {
          mma16816_p(acc[nt], xa.x, xb.x, xa.y, xb.y, bw[u][nt].x, bw[u][nt].y);
          mma16816_p(acc[nt], xa.z, xb.z, xa.w, xb.w, bw[u][nt].z, bw[u][nt].w);
        }
      }
    }
  }
  // sum the warps' partial tiles: fragment element i of lane -> (m, n)
#pragma unroll
  for (int nt = 0; nt < NT; ++nt)
    *reinterpret_cast<float4*>(red + ((warp * NT + nt) * 32 + lane) * 4) =
        make_float4(acc[nt][0], acc[nt][1], acc[nt][2], acc[nt][3]);
  __syncthreads();
  for (int idx = threadIdx.x; idx < nt_used * 128; idx += blockDim.x) {
    const int nt = idx / 128, e = idx % 128, ln = e / 4, i = e % 4;
    float sum = 0.f;
#pragma unroll
    for (int w = 0; w < kDecWarps; ++w) sum += red[((w * NT + nt) * 32 + ln) * 4 + i];
    const int m = (ln >> 2) + 8 * (i >> 1), n = 2 * (ln & 3) + (i & 1);
    fin[(nt * 16 + m) * 8 + n] = sum;
  }
  __syncthreads();
  // (alpha/r) (x A^T) B^T, RoPE, store: thread per (row m, channel i)
  const int m = threadIdx.x >> 3, i = threadIdx.x & 7;
  if (m < M) {
    float y1 = fin[(0 * 16 + m) * 8 + i], y2 = fin[(1 * 16 + m) * 8 + i];
    if (r > 0) {
      const __nv_bfloat16* Bm = reinterpret_cast<const __nv_bfloat16*>(p.bm[proj]);
      const __nv_bfloat16* b1 = Bm + ((int64_t)head * D + c0 + i) * r;
      const __nv_bfloat16* b2 = Bm + ((int64_t)head * D + half + c0 + i) * r;
      for (int j0 = 0; j0 < r; j0 += 8) {
        const uint4 u1 = __ldg(reinterpret_cast<const uint4*>(b1 + j0));
        const uint4 u2 = __ldg(reinterpret_cast<const uint4*>(b2 + j0));
        const __nv_bfloat16* e1 = reinterpret_cast<const __nv_bfloat16*>(&u1);
        const __nv_bfloat16* e2 = reinterpret_cast<const __nv_bfloat16*>(&u2);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const int j = j0 + e;
          const float uu = fin[((2 + j / 8) * 16 + m) * 8 + (j & 7)] * p.alpha_over_r;
          y1 += uu * __bfloat162float(e1[e]);
          y2 += uu * __bfloat162float(e2[e]);
        }
      }
    }
    const int b = m / p.L, l = m % p.L;
    const int c = c0 + i;
    if (proj < 2 && p.rope_base > 0.f) {
      const int pos = p.pos0 + pos_of(p.pos_dev, p.pos_stride, b) + l;
      float cs, sn;
      rope_cos_sin(pos, p.theta_hi[c], p.theta_lo[c], &cs, &sn);
      const float o1 = y1 * cs - y2 * sn, o2 = y2 * cs + y1 * sn;
      y1 = o1;
      y2 = o2;
    }
    const int H = proj == 0 ? p.Hq : p.Hkv;
    __nv_bfloat16* out = reinterpret_cast<__nv_bfloat16*>(p.out[proj]);
    const int64_t base = (((int64_t)b * H + head) * p.L + l) * D;
    out[base + c] = __float2bfloat16_rn(y1);
    out[base + c + half] = __float2bfloat16_rn(y2);
  }
  __syncthreads();                                          // shared memory reusable
}

__host__ __device__ inline size_t proj_decode_smem_bytes(int M16, int NT, int d_in) {
  return (size_t)M16 * d_in * 2 + (size_t)kDecWarps * NT * 128 * 4 + (size_t)NT * 128 * 4;
}

}  // namespace pdec
}  // namespace kvq
