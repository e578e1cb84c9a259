// One decode step of one layer as a single cooperative kernel: the LoRA Q/K/V
// projection of the new token (Section 3, Eq. 1 and the LoRA update),
// quantize-and-append of its key and value (Section 3.1), and split-K decode
// attention over the stored reconstruction (Sections 3.2-3.3).
//
// A decode step moves a few MB (the projection weights and the packed cache)
// and computes almost nothing, so its time is latency: the kernel starts every
// copy that depends on nothing in this step at entry, and CTAs hand results to
// one another only through tagged words (a float and the launch's tag in one
// 64-bit access; the reader polls until the tag is this launch's), one round
// trip per handoff, with no grid-wide barrier.  One CTA per SM (cooperative
// launch, so all CTAs are resident while some poll others' results):
//
//   entry    each warp issues TMA bulk copies of its projection units (8
//            stacked weight rows x 1024, 512 or 256 input channels) into a ring of
//            shared slots; one thread issues the first chunks of this CTA's
//            attention split (codes of the tokens already stored); the LoRA
//            up-projections are prefetched into L2; x goes to shared memory.
//   phase 1  per unit one 16x8 output tile on mma.sync; the partial goes to
//            the workspace as tagged words (deterministic slots).  The
//            stacked rows are [W_qkv; A_q; A_k; A_v], so the LoRA
//            down-projections ride along with the base GEMV.
//   phase 2  per attention item (split, kv head, sequence): pairs of query
//            heads per warp poll the unit partials of their channels, add
//            (alpha/r) U B^T and RoPE, and keep the bf16 queries in shared
//            memory (split 0 also stores them); the CTA whose split holds the
//            new token finishes its key and value the same way, stores them,
//            codes them into the cache and into the prefetched chunk.
//   phase 3  the split's attention; its partial goes out as tagged words and
//            the CTA holding the new token polls them and merges.
//
// The last CTA to finish (an arrival counter in the cache's device state)
// advances the token count and the launch epoch.  Every poll is bounded; a
// timeout sets the library's error word.
#include "decode_attn.cuh"
#include "proj_decode.cuh"

namespace kvq {
namespace {

constexpr int kWarpsF = 8;                   // warps per CTA
constexpr int kMaxSlots = 32;
constexpr size_t kSmemBudget = 227 * 1024 - 8192;   // dynamic shared memory (static kept aside)
// A projection unit is 8 stacked rows x ks input channels (ks = 1024 when
// d_in allows, else 512 or 256: fewer K slices mean fewer partials to hand
// over per output); its rows sit in shared memory at a stride of
// 2 ks + 64 bytes, so that the 16-byte operand loads of two rows in one
// quarter-warp fall on different banks.
__host__ __device__ constexpr int unit_bytes(int ks) { return 8 * (2 * ks + 64); }

struct StepArgs {
  const __nv_bfloat16* x;      // [B][d_in]
  const __nv_bfloat16* w;      // [n_out][d_in], n_out = (Hq + 2 Hkv) D
  const __nv_bfloat16* a[3];   // LoRA down-projections [r_p][d_in]
  const __nv_bfloat16* bm[3];  // LoRA up-projections [d_out_p][r_p]
  int r[3];
  __nv_bfloat16* out[3];       // q [B][Hq][1][D], k and v [B][Hkv][1][D]
  __nv_bfloat16* o;            // attention output [B][Hq][1][D]
  int d_in, n_out, ks, S, units;   // S = d_in / ks; units = (stacked rows / 8) * S
  int nslot, splits;
  int64_t part_off;            // unit partials: tagged words after the split partials
  int att_off, xs_off, xstride, q_off;   // shared memory layout (bytes)
  int bm_off, bm_bytes[3];     // staged LoRA up-projection rows (bytes; 0: read from global)
  float alpha_over_r, rope_base, scale;
  float theta_hi[128], theta_lo[128];
  int* err;
  Geom g;
};

__device__ __forceinline__ void mma_bf16(float c[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};\n"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Row n of the stacked matrix [W_qkv; A_q; A_k; A_v].
__device__ __forceinline__ const __nv_bfloat16* stacked_row(const StepArgs& a, int n) {
  if (n < a.n_out) return a.w + (int64_t)n * a.d_in;
  n -= a.n_out;
  for (int p = 0; p < 3; ++p) {
    if (n < a.r[p]) return a.a[p] + (int64_t)n * a.d_in;
    n -= a.r[p];
  }
  return a.w;   // not reached: units cover the stacked rows exactly
}

// Copies of unit u (8 rows x ks channels) into one slot; called by a whole
// warp, lanes 0..7 copy one row each.
__device__ __forceinline__ void issue_unit(const StepArgs& a, int u, unsigned char* slot,
                                           uint64_t* bar, int lane) {
  const int rowb = 2 * a.ks;
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  if (lane == 0) dattn::mbar_expect_tx(bar, 8 * rowb);
  __syncwarp();
  if (lane < 8) {
    const int tile = u / a.S, s = u % a.S;
    dattn::bulk_g2s(slot + lane * (rowb + 64), stacked_row(a, tile * 8 + lane) + s * a.ks, rowb,
                    bar);
  }
}

// Output channels of up to two stacked heads (0..Hq-1 queries, then keys,
// then values) of sequence b, worked on together by one warp so that their
// load latencies overlap: the sum of the unit partials, plus (alpha/r) U B^T,
// then RoPE for queries and keys.  Lane l holds channels l + 32 j
// (j < D/32); RoPE pairs are (j, j + D/64).  ush: 128 floats of shared
// scratch for this warp (the rank vectors U).
// bsrc[p] / brow0[p]: where row brow0[p] of B_p starts (shared memory when
// staged, else the global matrix with brow0 = 0).
template <int D>
__device__ void heads_values(const StepArgs& a, int b, const int (&hh)[2], int nh, int T0,
                             const uint64_t* __restrict__ part, uint32_t tag, float* ush,
                             const __nv_bfloat16* const (&bsrc)[3], const int (&brow0)[3],
                             float (&y)[2][D / 32]) {
  const Geom& g = a.g;
  const int lane = threadIdx.x & 31;
  constexpr int NJ = D / 32;
  constexpr int RB = D == 64 ? 2 : 1;       // B^T words per channel held in registers
  const int Hq = g.Hq, Hkv = g.H, M = g.B, S = a.S;
  int proj[2], head[2], r[2], arow[2];
  const __nv_bfloat16* bbase[2];     // B^T row of (head, channel 0) for each head
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int x = h < nh ? hh[h] : hh[0];
    proj[h] = x < Hq ? 0 : x < Hq + Hkv ? 1 : 2;
    head[h] = proj[h] == 0 ? x : proj[h] == 1 ? x - Hq : x - Hq - Hkv;
    const int rp = proj[h] == 0 ? a.r[0] : proj[h] == 1 ? a.r[1] : a.r[2];
    r[h] = h < nh ? rp : 0;
    arow[h] = a.n_out + (proj[h] >= 1 ? a.r[0] : 0) + (proj[h] >= 2 ? a.r[1] : 0);
    const __nv_bfloat16* src = proj[h] == 0 ? bsrc[0] : proj[h] == 1 ? bsrc[1] : bsrc[2];
    const int row0 = proj[h] == 0 ? brow0[0] : proj[h] == 1 ? brow0[1] : brow0[2];
    bbase[h] = src + ((int64_t)head[h] * D - row0) * rp;
  }
  auto part_at = [&](int n, int s) {
    return part + ((int64_t)((n >> 3) * S + s) * M + b) * 8 + (n & 7);
  };
  // B^T rows of the LoRA up-projection (first 16 ranks), issued first
  uint4 bw[2][NJ][RB];
#pragma unroll
  for (int h = 0; h < 2; ++h)
#pragma unroll
    for (int j = 0; j < NJ; ++j)
#pragma unroll
      for (int q = 0; q < RB; ++q) {
        bw[h][j][q] = make_uint4(0, 0, 0, 0);
        if (8 * q < r[h])
          bw[h][j][q] = *reinterpret_cast<const uint4*>(bbase[h] + (lane + 32 * j) * r[h] + 8 * q);
      }
  // partial sums over the S slices and the rank vectors U, in blocks of
  // four slices whose words are all loaded before any is used; a block is
  // reloaded until every word carries this launch's tag
  float u[2][2];
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    u[h][0] = u[h][1] = 0.f;
#pragma unroll
    for (int j = 0; j < NJ; ++j) y[h][j] = 0.f;
  }
  constexpr int SB = D == 64 ? 4 : 2;
  for (int s0 = 0; s0 < S; s0 += SB) {
    uint64_t wy[2][NJ][SB], wu[2][2][SB];
    for (long it = 0;; ++it) {
#pragma unroll
      for (int k = 0; k < SB; ++k)
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int s = s0 + k;
          const bool live = s < S && h < nh;
#pragma unroll
          for (int j = 0; j < NJ; ++j)
            wy[h][j][k] = live ? dattn::ld_tagged(part_at(hh[h] * D + lane + 32 * j, s)) : 0;
          wu[h][0][k] = live && lane < r[h] ? dattn::ld_tagged(part_at(arow[h] + lane, s)) : 0;
          wu[h][1][k] = live && lane + 32 < r[h] ? dattn::ld_tagged(part_at(arow[h] + lane + 32, s))
                                                 : 0;
        }
      bool ok = true;
#pragma unroll
      for (int k = 0; k < SB; ++k)
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          if (s0 + k >= S || h >= nh) continue;
#pragma unroll
          for (int j = 0; j < NJ; ++j) ok = ok && dattn::tag_is(wy[h][j][k], tag);
          if (lane < r[h]) ok = ok && dattn::tag_is(wu[h][0][k], tag);
          if (lane + 32 < r[h]) ok = ok && dattn::tag_is(wu[h][1][k], tag);
        }
      if (__all_sync(0xffffffffu, ok)) break;
      if (it > dattn::kPollLimit) {
        if (lane == 0) atomicOr(a.err, 16);
        break;
      }
    }
#pragma unroll
    for (int k = 0; k < SB; ++k)
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        if (s0 + k >= S || h >= nh) continue;
#pragma unroll
        for (int j = 0; j < NJ; ++j) y[h][j] += dattn::tagged_value(wy[h][j][k]);
        if (lane < r[h]) u[h][0] += dattn::tagged_value(wu[h][0][k]);
        if (lane + 32 < r[h]) u[h][1] += dattn::tagged_value(wu[h][1][k]);
      }
  }
  // U to shared memory, pre-scaled by alpha/r, read back as broadcasts
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    ush[h * 64 + lane] = u[h][0] * a.alpha_over_r;
    ush[h * 64 + 32 + lane] = u[h][1] * a.alpha_over_r;
  }
  __syncwarp();
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    if (r[h] == 0) continue;
#pragma unroll
    for (int j = 0; j < NJ; ++j) {
      auto rank8 = [&](const uint4& w8, int j0) {
        const __nv_bfloat16* e8 = reinterpret_cast<const __nv_bfloat16*>(&w8);
        const float4 ua = *reinterpret_cast<const float4*>(ush + h * 64 + j0);
        const float4 ub = *reinterpret_cast<const float4*>(ush + h * 64 + j0 + 4);
        y[h][j] += ua.x * __bfloat162float(e8[0]);
        y[h][j] += ua.y * __bfloat162float(e8[1]);
        y[h][j] += ua.z * __bfloat162float(e8[2]);
        y[h][j] += ua.w * __bfloat162float(e8[3]);
        y[h][j] += ub.x * __bfloat162float(e8[4]);
        y[h][j] += ub.y * __bfloat162float(e8[5]);
        y[h][j] += ub.z * __bfloat162float(e8[6]);
        y[h][j] += ub.w * __bfloat162float(e8[7]);
      };
#pragma unroll
      for (int q = 0; q < RB; ++q)
        if (8 * q < r[h]) rank8(bw[h][j][q], 8 * q);
      const __nv_bfloat16* brow = bbase[h] + (lane + 32 * j) * r[h];
      for (int j0 = 8 * RB; j0 < r[h]; j0 += 8)
        rank8(*reinterpret_cast<const uint4*>(brow + j0), j0);
    }
  }
  __syncwarp();                             // ush may be rewritten by the next call
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    if (h >= nh || proj[h] == 2 || !(a.rope_base > 0.f)) continue;
#pragma unroll
    for (int j = 0; j < NJ / 2; ++j) {
      const int c = lane + 32 * j;
      float cs, sn;
      pdec::rope_cos_sin(T0, a.theta_hi[c], a.theta_lo[c], &cs, &sn);
      const float y1 = y[h][j], y2 = y[h][j + NJ / 2];
      y[h][j] = y1 * cs - y2 * sn;
      y[h][j + NJ / 2] = y2 * cs + y1 * sn;
    }
  }
}

// Round to bf16, store at dst (lane l: channels l + 32 j), return the values.
template <int NJ>
__device__ __forceinline__ void store_bf16(const float* y, __nv_bfloat16* dst, float (&v)[NJ]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int j = 0; j < NJ; ++j) {
    const __nv_bfloat16 hb = __float2bfloat16_rn(y[j]);
    if (dst) dst[lane + 32 * j] = hb;
    v[j] = __bfloat162float(hb);
  }
}

// Code token t of (b, h) for keys (which = 0) or values into the cache; with
// `stage` also into row rr of that shared chunk copy.  Group j = channels
// 32 j .. 32 j + 31, i.e. value j of every lane.
template <int D, int BITS, int FMT>
__device__ void pack_token(const Geom& g, int which, int b, int h, int t, const float (&v)[D / 32],
                           unsigned char* stage, int rr) {
  using C = dattn::Cfg<D, BITS, FMT>;
  constexpr int NJ = D / 32, NG = C::NG;
  constexpr bool sym = FMT == KVQ_FMT_SYMMETRIC;
  const int lane = threadIdx.x & 31;
  const int P_CODES = which ? KVQ_PLANE_V_CODES : KVQ_PLANE_K_CODES;
  const int P_SCALE = which ? KVQ_PLANE_V_SCALE : KVQ_PLANE_K_SCALE;
  const int P_ZERO = which ? KVQ_PLANE_V_ZERO : KVQ_PLANE_K_ZERO;
  uint8_t* crow = plane_ptr<uint8_t>(g, P_CODES, b, h, t);
  unsigned char* srow = stage ? stage + (which ? C::VC_OFF : C::KC_OFF) + rr * C::CODE_B : nullptr;
  __half* ssc = stage ? reinterpret_cast<__half*>(stage + (which ? C::VS_OFF : C::KS_OFF)) + rr * NG
                      : nullptr;
  __half* sze = stage ? reinterpret_cast<__half*>(stage + (which ? C::VZ_OFF : C::KZ_OFF)) + rr * NG
                      : nullptr;
#pragma unroll
  for (int j = 0; j < NJ; ++j) {
    float lo = v[j], hi = sym ? fabsf(v[j]) : v[j];
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      if (sym) {
        hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, off));
      } else {
        lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, off));
        hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, off));
      }
    }
    uint32_t code;
    float s;
    if (sym) {
      const float qmax = (float)((1 << (BITS - 1)) - 1);
      s = fmaxf(__fdiv_rn(hi, qmax), 1e-8f);
      float q = rintf(__fdiv_rn(v[j], s));
      q = fminf(fmaxf(q, -qmax), qmax);
      code = (uint32_t)((int)q + (1 << (BITS - 1)));
    } else {
      const float cmax = (float)((1 << BITS) - 1);
      s = fmaxf(__fdiv_rn(__fsub_rn(hi, lo), cmax), 1e-8f);
      float c = rintf(__fdiv_rn(__fsub_rn(v[j], lo), s));
      c = fminf(fmaxf(c, 0.f), cmax);
      code = (uint32_t)c;
    }
    // 8 consecutive channels share one word, lowest channel in the low bits
    uint32_t word = code << (BITS * (lane & 7));
    word |= __shfl_xor_sync(0xffffffffu, word, 1);
    word |= __shfl_xor_sync(0xffffffffu, word, 2);
    word |= __shfl_xor_sync(0xffffffffu, word, 4);
    if ((lane & 7) == 0) {
      const int w8 = (32 * j + lane) >> 3;
      if (BITS == 4) {
        reinterpret_cast<uint32_t*>(crow)[w8] = word;
        if (srow) reinterpret_cast<uint32_t*>(srow)[w8] = word;
      } else {
        reinterpret_cast<uint16_t*>(crow)[w8] = (uint16_t)word;
        if (srow) reinterpret_cast<uint16_t*>(srow)[w8] = (uint16_t)word;
      }
    }
    if (lane == 0) {
      const __half hs = __float2half_rn(s), hz = __float2half_rn(lo + 0.0f);
      *plane_ptr<__half>(g, P_SCALE, b, h, t, j) = hs;
      if (ssc) ssc[j] = hs;
      if (!sym) {
        *plane_ptr<__half>(g, P_ZERO, b, h, t, j) = hz;
        if (sze) sze[j] = hz;
      }
    }
  }
}

template <int D, int BITS, int FMT, int AST>
__global__ void __launch_bounds__(kWarpsF * 32, 1)
decode_step_kernel(const __grid_constant__ StepArgs a) {
  extern __shared__ __align__(1024) unsigned char sm[];
  __shared__ uint64_t ubar[kMaxSlots];
  __shared__ uint64_t abar[AST];
  __shared__ uint64_t bbar;
  __shared__ uint64_t xbar;
  __shared__ __align__(16) float ush[kWarpsF][128];
  const Geom& g = a.g;
  CacheState* st = g.state;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gid = lane >> 2, tid = lane & 3;
  // ---- before the dependency wait: read-only inputs only (weights) ---------
  // The weight units and the LoRA up-projection rows do not depend on the
  // preceding kernel on the stream, so their copies start while it drains
  // (programmatic dependent launch); everything else waits for it.
  if (threadIdx.x == 0) {
    for (int i = 0; i < a.nslot; ++i) dattn::mbar_init(&ubar[i], 1);
    dattn::mbar_init(&bbar, 1);
    dattn::mbar_init(&xbar, 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();
  const int u_begin = (int)((int64_t)blockIdx.x * a.units / gridDim.x);
  const int n_local = (int)((int64_t)(blockIdx.x + 1) * a.units / gridDim.x) - u_begin;
  const int unitb = unit_bytes(a.ks), rstride = 2 * a.ks + 64;
  unsigned char* ring = sm;
  for (int i = warp; i < min(n_local, a.nslot); i += kWarpsF)
    issue_unit(a, u_begin + i, ring + (i % a.nslot) * unitb, &ubar[i % a.nslot], lane);
  const int items3 = a.splits * g.H * g.B;
  const int grp = g.Hq / g.H;
  // LoRA up-projection rows of this CTA's first item (its kv head's query
  // heads, key and value) into shared memory
  const bool staged = a.bm_off > 0 && (int)blockIdx.x < items3;
  if (staged && threadIdx.x == 0) {
    const int hkv0 = (blockIdx.x / a.splits) % g.H;
    dattn::mbar_expect_tx(&bbar, a.bm_bytes[0] + a.bm_bytes[1] + a.bm_bytes[2]);
    unsigned char* dst = sm + a.bm_off;
    const int64_t first_row[3] = {(int64_t)hkv0 * grp * D, (int64_t)hkv0 * D, (int64_t)hkv0 * D};
    for (int p = 0; p < 3; ++p) {
      if (a.bm_bytes[p])
        dattn::bulk_g2s(dst, a.bm[p] + first_row[p] * a.r[p], a.bm_bytes[p], &bbar);
      dst += a.bm_bytes[p];
    }
  }
  if (threadIdx.x < 3) {                   // LoRA up-projections -> L2, a share per CTA
    const int p = threadIdx.x;
    const int d_out = (p == 0 ? g.Hq : g.H) * D;
    const int64_t bytes = (int64_t)d_out * a.r[p] * 2;  // a multiple of 16
    const int64_t lo = bytes * blockIdx.x / gridDim.x / 16 * 16;
    const int64_t hi = bytes * (blockIdx.x + 1) / gridDim.x / 16 * 16;
    if (hi > lo)
      asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;"
                   ::"l"(reinterpret_cast<const char*>(a.bm[p]) + lo), "r"((uint32_t)(hi - lo))
                   : "memory");
  }
  pdl_trigger();
  pdl_wait();

  // x (the step's input, written by the preceding kernel) to shared memory:
  // one bulk copy per row, in flight with the token-count read below
  unsigned char* xs = sm + a.xs_off;
  const int M = g.B;
  const bool x_bulk = (reinterpret_cast<uintptr_t>(a.x) & 15) == 0;
  if (x_bulk && threadIdx.x == 0) {
    dattn::mbar_expect_tx(&xbar, (uint32_t)(M * 2 * a.d_in));
    for (int m = 0; m < M; ++m)
      dattn::bulk_g2s(xs + m * a.xstride, a.x + (int64_t)m * a.d_in, 2 * a.d_in, &xbar);
  }
  // tokens before this step and the launch epoch: read once (thread 0) and
  // shared, so that both reads are complete before this CTA arrives on the
  // counter below
  __shared__ int s_T0;
  __shared__ uint32_t s_epoch;
  if (threadIdx.x == 0) {
    s_T0 = *reinterpret_cast<volatile int32_t*>(&st->tokens);
    s_epoch = *reinterpret_cast<volatile uint32_t*>(g.epoch);
  }
  __syncthreads();
  const int T0 = s_T0;
  const uint32_t epoch = s_epoch;
  const uint32_t tag = 0xFFC00000u | ((epoch + 1) & 0x003FFFFFu);   // a NaN no arithmetic makes
  const bool room = T0 >= 0 && T0 + 1 <= g.Tmax;
  const int T = T0 + 1;
  unsigned char* asmem = sm + a.att_off;
  uint64_t* part = reinterpret_cast<uint64_t*>(g.pl[KVQ_PLANE_WORKSPACE].p) + a.part_off;
  const bool attend_here = room && (int)blockIdx.x < items3;
  int early = 0;                           // attention chunks issued ahead of the split
  if (attend_here) {
    const int rest = blockIdx.x / a.splits;
    const dattn::SplitPlan sp = dattn::split_plan<FMT>(g, T, a.splits, blockIdx.x % a.splits);
    dattn::split_prologue<D, BITS, FMT, AST>(g, rest / g.H, rest % g.H, sp, asmem, abar);
    early = min(AST, sp.nchunks);
  }
  if (x_bulk) {
    if (threadIdx.x == 0 && !dattn::mbar_wait(&xbar, 0)) atomicOr(a.err, 1);
  } else {                                 // x not 16-byte aligned: element loads
    for (int i = threadIdx.x; i < M * a.d_in; i += blockDim.x) {
      const int m = i / a.d_in, k = i - m * a.d_in;
      *reinterpret_cast<__nv_bfloat16*>(xs + m * a.xstride + 2 * k) = a.x[i];
    }
  }
  __syncthreads();
  // Every CTA has read the token count and the epoch once it arrives here;
  // the last to arrive advances both (the values this launch uses stay in
  // registers).  One thread of the last warp, while the units are landing.
  if (threadIdx.x == 32 * (kWarpsF - 1)) {
    __threadfence();
    const unsigned prev = atomicAdd(reinterpret_cast<unsigned*>(&st->pad[2]), 1u);
    if (prev == gridDim.x - 1) {
      st->pad[2] = 0;
      if (room) st->tokens = T;
      *reinterpret_cast<volatile uint32_t*>(g.epoch) = epoch + 1;
    }
  }

  // ---- phase 1: unit partials ---------------------------------------------
  int i = warp;
  bool ok1 = true;
  for (; i < n_local; i += kWarpsF) {
    const int slot = i % a.nslot;
    if (!dattn::mbar_wait(&ubar[slot], (i / a.nslot) & 1)) {
      ok1 = false;
      break;
    }
    const int u = u_begin + i, tile = u / a.S, s = u % a.S;
    const unsigned char* sl = ring + slot * unitb;
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 8
    for (int j = 0; j < a.ks / 32; ++j) {
      // thread (gid, tid) holds channels 8 tid .. 8 tid + 7 of the 32-channel
      // chunk j; words .x/.y feed the first k-step and .z/.w the second
      const int k = s * a.ks + 32 * j + 8 * tid;
      uint4 xa = make_uint4(0, 0, 0, 0), xb = make_uint4(0, 0, 0, 0);
      if (gid < M) xa = *reinterpret_cast<const uint4*>(xs + gid * a.xstride + 2 * k);
      if (gid + 8 < M) xb = *reinterpret_cast<const uint4*>(xs + (gid + 8) * a.xstride + 2 * k);
      const uint4 bw = *reinterpret_cast<const uint4*>(sl + gid * rstride + 64 * j + 16 * tid);
      mma_bf16(acc, xa.x, xb.x, xa.y, xb.y, bw.x, bw.y);
      mma_bf16(acc, xa.z, xb.z, xa.w, xb.w, bw.z, bw.w);
    }
    uint64_t* pp = part + (int64_t)(tile * a.S + s) * M * 8;
    if (gid < M) {
      dattn::st_tagged(pp + gid * 8 + 2 * tid, acc[0], tag);
      dattn::st_tagged(pp + gid * 8 + 2 * tid + 1, acc[1], tag);
    }
    if (gid + 8 < M) {
      dattn::st_tagged(pp + (gid + 8) * 8 + 2 * tid, acc[2], tag);
      dattn::st_tagged(pp + (gid + 8) * 8 + 2 * tid + 1, acc[3], tag);
    }
    __syncwarp();
    if (i + a.nslot < n_local) issue_unit(a, u + a.nslot, ring + slot * unitb, &ubar[slot], lane);
  }
  if (!ok1) {                              // flag, then let this warp's copies land
    if (lane == 0) {
      atomicOr(a.err, 8);
      for (int j = i; j < min(n_local, i + a.nslot); j += kWarpsF)
        dattn::mbar_wait(&ubar[j % a.nslot], (j / a.nslot) & 1);
    }
    __syncwarp();
  }

  // ---- phases 2 and 3, per attention item ------------------------------------
  constexpr int NJ = D / 32;
  __nv_bfloat16* qsm = reinterpret_cast<__nv_bfloat16*>(sm + a.q_off);   // [grp][D]
  for (int it = blockIdx.x; it < items3; it += gridDim.x) {
    const int split = it % a.splits, rest = it / a.splits;
    const int hkv = rest % g.H, b = rest / g.H;
    const __nv_bfloat16* bsrc[3] = {a.bm[0], a.bm[1], a.bm[2]};
    int brow0[3] = {0, 0, 0};
    if (staged && it == (int)blockIdx.x) {
      bool landed = dattn::mbar_wait(&bbar, 0);
      if (!landed) {
        if (threadIdx.x == 0) atomicOr(a.err, 1);
      } else {
        const unsigned char* src = sm + a.bm_off;
        for (int p = 0; p < 3; ++p) {
          bsrc[p] = reinterpret_cast<const __nv_bfloat16*>(src);
          brow0[p] = p == 0 ? hkv * grp * D : hkv * D;
          src += a.bm_bytes[p];
        }
      }
    }
    const dattn::SplitPlan sp = dattn::split_plan<FMT>(g, T, a.splits, split);
    if (it != (int)blockIdx.x && room) {
      dattn::split_prologue<D, BITS, FMT, AST>(g, b, hkv, sp, asmem, abar);
      early = min(AST, sp.nchunks);
    }
    const bool kv_here = sp.ts <= T0 && T0 < sp.te;     // this split holds the new token
    const int nfin = grp + (kv_here ? 2 : 0);           // query heads, then key and value
    for (int f0 = 2 * warp; f0 < nfin; f0 += 2 * kWarpsF) {
      const int nh = min(2, nfin - f0);
      int hh[2];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int f = min(f0 + h, nfin - 1);
        hh[h] = f < grp ? hkv * grp + f : g.Hq + (f - grp) * g.H + hkv;
      }
      float y[2][NJ];
      heads_values<D>(a, b, hh, nh, T0, part, tag, ush[warp], bsrc, brow0, y);
      for (int h = 0; h < nh; ++h) {
        const int f = f0 + h;
        float v[NJ];
        if (f < grp) {
          store_bf16<NJ>(y[h], split == 0 ? a.out[0] + ((int64_t)b * g.Hq + hh[h]) * D : nullptr,
                         v);
#pragma unroll
          for (int j = 0; j < NJ; ++j) qsm[f * D + lane + 32 * j] = __float2bfloat16_rn(v[j]);
        } else {
          const int which = f - grp;                     // 0 keys, 1 values
          store_bf16<NJ>(y[h], a.out[1 + which] + ((int64_t)b * g.H + hkv) * D, v);
          if (room) {
            // the chunk holding the token was copied at entry (before the
            // token existed): once it has landed, overwrite the token's row
            const int ci = (T0 - sp.ts) / dattn::kCT;
            unsigned char* stage = nullptr;
            if (ci < early) {
              bool landed = true;
              if (lane == 0) landed = dattn::mbar_wait(&abar[ci % AST], (ci / AST) & 1);
              landed = __shfl_sync(0xffffffffu, landed, 0);
              if (landed) stage = asmem + (ci % AST) * dattn::Cfg<D, BITS, FMT>::STAGE_B;
              else if (lane == 0) atomicOr(a.err, 1);
            }
            pack_token<D, BITS, FMT>(g, which, b, hkv, T0, v, stage,
                                     T0 - sp.ts - ci * dattn::kCT);
          }
        }
      }
    }
    __syncthreads();
    if (room)
      dattn::decode_split<D, BITS, FMT, AST, kWarpsF>(g, qsm, a.scale, a.err, a.o, split,
                                                      a.splits, a.splits, hkv, b, T, asmem, abar,
                                                      true, tag, kv_here);
  }
}

template <int D>
constexpr int att_stages() {
  return D == 64 ? 8 : 4;
}

// Shared memory and workspace plan; false if the fused kernel cannot hold it.
bool plan_step(const Geom& g, int d_in, const int r[3], size_t att_bytes, StepArgs* a,
               size_t* smem) {
  const int n_out = (g.Hq + 2 * g.H) * g.D;
  const int rows = n_out + r[0] + r[1] + r[2];
  const int ks = d_in % 1024 == 0 ? 1024 : d_in % 512 == 0 ? 512 : 256;
  const int S = d_in / ks;
  const int units = rows / 8 * S;
  const int grid = num_sms();
  const int per_cta = (units + grid - 1) / grid;
  const size_t att = (att_bytes + 127) / 128 * 128;
  const int xstride = d_in * 2 + 64;
  const size_t xs = (size_t)g.B * xstride;
  const size_t qs = (size_t)(g.Hq / g.H) * g.D * 2;
  const int bmb[3] = {(g.Hq / g.H) * g.D * r[0] * 2, g.D * r[1] * 2, g.D * r[2] * 2};
  size_t bms = (size_t)bmb[0] + bmb[1] + bmb[2];
  if (att + xs + qs + bms + (size_t)kWarpsF * unit_bytes(ks) > kSmemBudget) bms = 0;
  if (att + xs + qs >= kSmemBudget) return false;
  int nslot = (int)((kSmemBudget - att - xs - qs - bms) / unit_bytes(ks));
  nslot = min(nslot, kMaxSlots) / kWarpsF * kWarpsF;
  nslot = min(nslot, (per_cta + kWarpsF - 1) / kWarpsF * kWarpsF);
  if (nslot < kWarpsF) return false;
  // workspace, in tagged 64-bit words: split partials [B][Hq][splits][D + 2],
  // then the unit partials [rows / 8][S][B][8]
  int splits = grid / (g.B * g.H);
  splits = splits < 1 ? 1 : splits > 16 ? 16 : splits;
  auto words = [&](int sp) {
    return (size_t)g.B * g.Hq * sp * (g.D + kWsStride) + (size_t)rows * S * g.B;
  };
  while (splits > 1 && 2 * words(splits) > workspace_floats(g)) --splits;
  if (2 * words(splits) > workspace_floats(g)) return false;
  const int64_t part_off = (int64_t)g.B * g.Hq * splits * (g.D + kWsStride);
  a->n_out = n_out;
  a->ks = ks;
  a->S = S;
  a->units = units;
  a->nslot = nslot;
  a->splits = splits;
  a->part_off = part_off;
  a->att_off = nslot * unit_bytes(ks);
  a->xs_off = a->att_off + (int)att;
  a->xstride = xstride;
  a->q_off = a->xs_off + (int)xs;
  a->bm_off = bms ? (int)((a->q_off + qs + 15) / 16 * 16) : 0;
  for (int p = 0; p < 3; ++p) a->bm_bytes[p] = bms ? bmb[p] : 0;
  *smem = bms ? (size_t)a->bm_off + bms : (size_t)a->q_off + qs;
  return true;
}

template <int D, int BITS, int FMT>
cudaError_t launch_step(StepArgs& a, const int r[3], cudaStream_t s) {
  constexpr int AST = att_stages<D>();
  size_t smem = 0;
  if (!plan_step(a.g, a.d_in, r, dattn::attn_smem_bytes<D, BITS, FMT, AST, kWarpsF>(), &a,
                 &smem))
    return cudaErrorNotSupported;
  auto kern = decode_step_kernel<D, BITS, FMT, AST>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  int per_sm = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kWarpsF * 32, smem);
  if (e != cudaSuccess) return e;
  if (per_sm < 1) return cudaErrorNotSupported;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(num_sms());
  cfg.blockDim = dim3(kWarpsF * 32);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  e = cudaLaunchKernelEx(&cfg, kern, a);
  if (e != cudaSuccess) {                  // without the early start
    (void)cudaGetLastError();
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, kern, a);
  }
  return e;
}

template <int D>
cudaError_t launch_fmt(StepArgs& a, const int r[3], cudaStream_t s) {
  const Geom& g = a.g;
  const bool sym = g.fmt == KVQ_FMT_SYMMETRIC;
  if (g.kb == 4) return sym ? launch_step<D, 4, KVQ_FMT_SYMMETRIC>(a, r, s)
                            : launch_step<D, 4, KVQ_FMT_AFFINE>(a, r, s);
  return sym ? launch_step<D, 2, KVQ_FMT_SYMMETRIC>(a, r, s)
             : launch_step<D, 2, KVQ_FMT_AFFINE>(a, r, s);
}

size_t att_bytes_for(const Geom& g) {
  if (g.D == 64) return g.kb == 4 ? dattn::attn_smem_bytes<64, 4, KVQ_FMT_AFFINE, 8, kWarpsF>()
                                  : dattn::attn_smem_bytes<64, 2, KVQ_FMT_AFFINE, 8, kWarpsF>();
  return g.kb == 4 ? dattn::attn_smem_bytes<128, 4, KVQ_FMT_AFFINE, 4, kWarpsF>()
                   : dattn::attn_smem_bytes<128, 2, KVQ_FMT_AFFINE, 4, kWarpsF>();
}

}  // namespace

// The fused step covers bf16 affine/symmetric caches with 2/4-bit codes,
// G = 32, head_dim 64/128, up to 16 sequences, d_in a multiple of 256 and
// LoRA ranks that are multiples of 8 up to 64, when its shared-memory plan
// fits one SM.
bool decode_step_supported(const Geom& g, int d_in, const int r[3]) {
  const bool fmt_ok = (g.fmt == KVQ_FMT_AFFINE || g.fmt == KVQ_FMT_SYMMETRIC) &&
                      g.act == KVQ_BF16 && g.G == 32 && g.kb == g.vb &&
                      (g.kb == 2 || g.kb == 4) && (g.D == 64 || g.D == 128);
  if (!fmt_ok || g.layout != KVQ_LAYOUT_UNIFORM || g.Hq / g.H > 16 || g.B > 16 || d_in <= 0 ||
      d_in % 256)
    return false;
  for (int p = 0; p < 3; ++p)
    if (r[p] < 0 || r[p] > 64 || r[p] % 8) return false;
  StepArgs a;
  size_t smem = 0;
  return plan_step(g, d_in, r, att_bytes_for(g), &a, &smem);
}

cudaError_t launch_decode_step(const Geom& g, const void* x, int d_in, const void* w,
                               const void* const a_[3], const void* const bm[3], const int r[3],
                               float alpha_over_r, float rope_base, float scale,
                               void* const qkv[3], void* out, int* err, cudaStream_t s) {
  StepArgs a;
  a.x = reinterpret_cast<const __nv_bfloat16*>(x);
  a.w = reinterpret_cast<const __nv_bfloat16*>(w);
  for (int i = 0; i < 3; ++i) {
    a.a[i] = reinterpret_cast<const __nv_bfloat16*>(a_[i]);
    a.bm[i] = reinterpret_cast<const __nv_bfloat16*>(bm[i]);
    a.r[i] = r[i];
    a.out[i] = reinterpret_cast<__nv_bfloat16*>(qkv[i]);
  }
  a.o = reinterpret_cast<__nv_bfloat16*>(out);
  a.d_in = d_in;
  a.alpha_over_r = alpha_over_r;
  a.rope_base = rope_base;
  a.scale = scale;
  rope_theta_table(rope_base, g.D, a.theta_hi, a.theta_lo);
  a.err = err;
  a.g = g;
  return g.D == 64 ? launch_fmt<64>(a, r, s) : launch_fmt<128>(a, r, s);
}

}  // namespace kvq
