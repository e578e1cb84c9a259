// One decode step of one layer as a single cooperative kernel: the LoRA Q/K/V
// projection of the new token (Section 3, Eq. 1 and Eq. lora), quantize-and-
// append of its key and value (Section 3.1), and split-K decode attention over
// the stored reconstruction (Sections 3.2-3.3).
//
// Launched with one CTA per SM (cooperative, so all CTAs are resident):
//   phase 1  projection pair-tiles, round-robin over the CTAs
//   barrier
//   phase 2  one warp per (sequence, kv head, key|value) codes the new token
//   barrier
//   phase 3  decode attention splits, round-robin; the last CTA of each
//            (sequence, kv head) merges the splits (arrival counter)
// The last CTA to finish phase 3 advances the cache's token count.  The grid
// barriers count arrivals and generations in the cache's device state; every
// wait is bounded and a timeout sets the library's error word.  Formats and
// shapes outside this path run as the three separate calls.
#include "decode_attn.cuh"
#include "proj_decode.cuh"

namespace kvq {
namespace {

constexpr long kBarrierLimit = 1L << 22;     // polls of ~0.1 us: about half a second

struct StepArgs {
  pdec::ProjArgs p;
  Geom g;
  float scale;
  int* err;
  __nv_bfloat16* out;
};

// Grid-wide barrier over the cache's state words pad[0] (arrivals) and
// pad[1] (generation).  Returns false (all threads) if the wait timed out.
__device__ bool grid_barrier(CacheState* st, int* err) {
  __shared__ int ok_sh;
  __syncthreads();
  if (threadIdx.x == 0) {
    volatile int32_t* gen = &st->pad[1];
    const int32_t my_gen = *gen;
    __threadfence();
    const unsigned arrived =
        atomicAdd(reinterpret_cast<unsigned*>(&st->pad[0]), 1u) + 1u;
    int ok = 1;
    if (arrived == gridDim.x) {
      st->pad[0] = 0;
      __threadfence();
      atomicAdd(reinterpret_cast<int*>(&st->pad[1]), 1);
    } else {
      long i = 0;
      while (*gen == my_gen) {
        if (++i > kBarrierLimit) {
          ok = 0;
          atomicOr(err, 4);
          break;
        }
        __nanosleep(64);
      }
    }
    __threadfence();
    ok_sh = ok;
  }
  __syncthreads();
  return ok_sh != 0;
}

// Code the new token t of (b, h) for keys (which = 0) or values: one warp,
// lane l < D/8 holds channels 8l .. 8l+7; groups of 32 channels are 4 lanes.
template <int D, int BITS>
__device__ void pack_token_warp(const Geom& g, const __nv_bfloat16* x, int which, int b, int h,
                                int t, bool sym) {
  const int lane = threadIdx.x & 31;
  const bool live = lane < D / 8;
  float v[8];
  const __nv_bfloat16* src = x + ((int64_t)b * g.H + h) * D + 8 * (live ? lane : 0);
  const uint4 u = *reinterpret_cast<const uint4*>(src);
  const __nv_bfloat162* p2 = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 f = __bfloat1622float2(p2[i]);
    v[2 * i] = f.x;
    v[2 * i + 1] = f.y;
  }
  float lo = v[0], hi = sym ? fabsf(v[0]) : v[0];
#pragma unroll
  for (int i = 1; i < 8; ++i) {
    if (sym) hi = fmaxf(hi, fabsf(v[i]));
    else { lo = fminf(lo, v[i]); hi = fmaxf(hi, v[i]); }
  }
  for (int off = 2; off > 0; off >>= 1) {          // 4 lanes per group of 32
    lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, off));
    hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, off));
  }
  if (!live) return;
  uint32_t word = 0;
  float s;
  if (sym) {
    const float qmax = (float)((1 << (BITS - 1)) - 1);
    s = fmaxf(__fdiv_rn(hi, qmax), 1e-8f);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      float q = rintf(__fdiv_rn(v[i], s));
      q = fminf(fmaxf(q, -qmax), qmax);
      word |= (uint32_t)((int)q + (1 << (BITS - 1))) << (i * BITS);
    }
  } else {
    const float cmax = (float)((1 << BITS) - 1);
    s = fmaxf(__fdiv_rn(__fsub_rn(hi, lo), cmax), 1e-8f);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      float c = rintf(__fdiv_rn(__fsub_rn(v[i], lo), s));
      c = fminf(fmaxf(c, 0.f), cmax);
      word |= (uint32_t)c << (i * BITS);
    }
  }
  const int P_CODES = which ? KVQ_PLANE_V_CODES : KVQ_PLANE_K_CODES;
  const int P_SCALE = which ? KVQ_PLANE_V_SCALE : KVQ_PLANE_K_SCALE;
  const int P_ZERO = which ? KVQ_PLANE_V_ZERO : KVQ_PLANE_K_ZERO;
  uint8_t* crow = plane_ptr<uint8_t>(g, P_CODES, b, h, t);
  if (BITS == 4) *reinterpret_cast<uint32_t*>(crow + 4 * lane) = word;
  else *reinterpret_cast<uint16_t*>(crow + 2 * lane) = (uint16_t)word;
  if ((lane & 3) == 0) {
    const int grp = lane / 4;
    *plane_ptr<__half>(g, P_SCALE, b, h, t, grp) = __float2half_rn(s);
    if (!sym) *plane_ptr<__half>(g, P_ZERO, b, h, t, grp) = __float2half_rn(lo + 0.0f);
  }
}

template <int M16, int NT, int D, int BITS, int FMT>
__global__ void __launch_bounds__(pdec::kDecWarps * 32, 1) decode_step_kernel(StepArgs a) {
  extern __shared__ __align__(1024) unsigned char sm[];
  __shared__ int last_sh;
  const Geom& g = a.g;
  const int T0 = cache_tokens(g);                  // tokens before this step
  const bool room = T0 + 1 <= g.Tmax;
  // ---- phase 1: projection ----
  const int tiles = (a.p.Hq + 2 * a.p.Hkv) * (a.p.D / 16);
  for (int t = blockIdx.x; t < tiles; t += gridDim.x) pdec::proj_decode_tile<M16, NT>(a.p, t, sm);
  if (!grid_barrier(g.state, a.err)) return;
  // ---- phase 2: code the new token ----
  if (room) {
    const int warps = gridDim.x * (blockDim.x / 32);
    const int items = g.B * g.H * 2;
    for (int it = blockIdx.x * (blockDim.x / 32) + (threadIdx.x >> 5); it < items; it += warps) {
      const int which = it & 1, bh = it >> 1;
      pack_token_warp<D, BITS>(g, reinterpret_cast<const __nv_bfloat16*>(a.p.out[1 + which]),
                               which, bh / g.H, bh % g.H, T0, FMT == KVQ_FMT_SYMMETRIC);
    }
  } else if (blockIdx.x == 0 && threadIdx.x == 0) {
    atomicOr(&g.state->error, kErrCapacity);
  }
  if (!grid_barrier(g.state, a.err)) return;
  if (!room) return;
  // ---- phase 3: attention over T0 + 1 tokens ----
  const int items = g.splits * g.H * g.B;
  for (int it = blockIdx.x; it < items; it += gridDim.x) {
    const int split = it % g.splits, rest = it / g.splits;
    dattn::decode_split<D, BITS, FMT>(g, reinterpret_cast<const __nv_bfloat16*>(a.p.out[0]),
                                      a.scale, a.err, a.out, split, rest % g.H, rest / g.H,
                                      T0 + 1, sm);
  }
  // ---- the last CTA out advances the token count ----
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    const unsigned prev = atomicAdd(reinterpret_cast<unsigned*>(&g.state->pad[2]), 1u);
    last_sh = prev == gridDim.x - 1;
    if (last_sh) {
      g.state->pad[2] = 0;
      g.state->tokens = T0 + 1;
      __threadfence();
    }
  }
}

template <int M16, int NT, int D, int BITS, int FMT>
cudaError_t launch_step(const StepArgs& a, cudaStream_t s) {
  auto kern = decode_step_kernel<M16, NT, D, BITS, FMT>;
  size_t smem = pdec::proj_decode_smem_bytes(M16, NT, a.p.d_in);
  const size_t sa = dattn::attn_smem_bytes<D, BITS, FMT>();
  if (sa > smem) smem = sa;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  int per_sm = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, pdec::kDecWarps * 32, smem);
  if (e != cudaSuccess) return e;
  if (per_sm < 1) return cudaErrorNotSupported;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(num_sms());
  cfg.blockDim = dim3(pdec::kDecWarps * 32);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, a);
}

template <int M16, int NT>
cudaError_t launch_fmt(const StepArgs& a, cudaStream_t s) {
  const Geom& g = a.g;
  if (g.D == 64) {
    if (g.kb == 4) return g.fmt == KVQ_FMT_SYMMETRIC ? launch_step<M16, NT, 64, 4, KVQ_FMT_SYMMETRIC>(a, s)
                                                     : launch_step<M16, NT, 64, 4, KVQ_FMT_AFFINE>(a, s);
    return g.fmt == KVQ_FMT_SYMMETRIC ? launch_step<M16, NT, 64, 2, KVQ_FMT_SYMMETRIC>(a, s)
                                      : launch_step<M16, NT, 64, 2, KVQ_FMT_AFFINE>(a, s);
  }
  if (g.kb == 4) return g.fmt == KVQ_FMT_SYMMETRIC ? launch_step<M16, NT, 128, 4, KVQ_FMT_SYMMETRIC>(a, s)
                                                   : launch_step<M16, NT, 128, 4, KVQ_FMT_AFFINE>(a, s);
  return g.fmt == KVQ_FMT_SYMMETRIC ? launch_step<M16, NT, 128, 2, KVQ_FMT_SYMMETRIC>(a, s)
                                    : launch_step<M16, NT, 128, 2, KVQ_FMT_AFFINE>(a, s);
}

}  // namespace

// The fused step covers bf16 affine/symmetric caches with 2/4-bit codes,
// G = 32, head_dim 64/128, up to 16 sequences and ranks up to 64.
bool decode_step_supported(const Geom& g, int d_in, const int r[3]) {
  const bool fmt_ok = (g.fmt == KVQ_FMT_AFFINE || g.fmt == KVQ_FMT_SYMMETRIC) &&
                      g.act == KVQ_BF16 && g.G == 32 && g.kb == g.vb &&
                      (g.kb == 2 || g.kb == 4) && (g.D == 64 || g.D == 128);
  const int grp = g.Hq / g.H;
  return fmt_ok && grp <= 16 && g.B <= 16 && d_in % 32 == 0 &&
         (size_t)16 * d_in * 2 <= 160 * 1024 && r[0] <= 64 && r[1] <= 64 && r[2] <= 64;
}

cudaError_t launch_decode_step(const Geom& g, const void* x, int d_in, const void* w,
                                   const void* const a_[3], const void* const bm[3],
                                   const int r[3], float alpha_over_r, float rope_base,
                                   float scale, void* const qkv[3], void* out, int* err,
                                   cudaStream_t s) {
  StepArgs a;
  pdec::ProjArgs& p = a.p;
  p.x = x;
  p.w = w;
  for (int i = 0; i < 3; ++i) {
    p.a[i] = a_[i];
    p.bm[i] = bm[i];
    p.r[i] = r[i];
    p.out[i] = qkv[i];
  }
  p.B = g.B; p.L = 1; p.d_in = d_in; p.Hq = g.Hq; p.Hkv = g.H; p.D = g.D; p.pos0 = 0;
  p.act = KVQ_BF16;
  p.pos_dev = &g.state->tokens;
  p.alpha_over_r = alpha_over_r;
  p.rope_base = rope_base;
  rope_theta_table(rope_base, g.D, p.theta_hi, p.theta_lo);
  a.g = g;
  a.scale = scale;
  a.err = err;
  a.out = reinterpret_cast<__nv_bfloat16*>(out);
  const int rmax = max(r[0], max(r[1], r[2]));
  const int nt = 2 + rmax / 8;
  if (g.B <= 8) return nt <= 4 ? launch_fmt<8, 4>(a, s) : launch_fmt<8, pdec::kDecMaxNt>(a, s);
  return nt <= 4 ? launch_fmt<16, 4>(a, s) : launch_fmt<16, pdec::kDecMaxNt>(a, s);
}

}  // namespace kvq
