// Streaming split-K decode attention over the packed cache (§3.1 cache
// formats, §3.2-3.3 attention over the stored reconstruction, L = 1).
//
// Persistent CTAs, one per SM: the (sequence, kv head, 32-token block) space
// is flattened head-major and cut into one contiguous range per CTA, so every
// CTA streams the same number of blocks whatever B, Hkv and T are.  One
// producer warp copies each block (codes and fp16 metadata) with
// cp.async.bulk into a deep ring of shared-memory stages (full/empty
// mbarriers, bounded waits); eight consumer warps take the ring's blocks in
// turn.  A warp keeps a running softmax state per kv head; where the CTA's
// range crosses into the next head, its warps hand their partials to a
// shared-memory slot, the last of them merges the slot, and where a head
// spans several CTAs the last CTA to finish it (an arrival counter) merges
// their partials from the workspace.  No CTA ever waits on another.
//
// Tensor-core layout (mma.sync m16n8k16): tokens are the MMA rows and the
// g = Hq / Hkv query heads of the kv head its columns, so GQA heads share
// every code that is unpacked.
//   scores   S^T[t][h] = sum_d k_hat[t][d] q[h][d]
//     A = key codes as exact bf16 integers (0x4300 | c) = 128 + c, B = q.
//     Per-token groups: one accumulator per group, then
//       S = sum_g s_tg acc_g + (m_tg - 128 s_tg) sum_{d in g} q_d.
//     KIVI keys (one scale per 32-token block and channel): B = q * s_blk as
//     bf16 high + low parts (two MMAs); the 128 of the codes is removed with
//     an MMA over a constant operand, and sum_d q_d m_d is added per block.
//   softmax  in base 2 with the softmax scale folded in; P goes to fp16 and
//     movmatrix transposes each 8x8 tile into the B operand of P V.
//   values   O^T[d][h] = sum_t v_hat[t][d] p[h][t]
//     A = value codes as exact fp16 integers (0x6400 | c) = 1024 + c,
//     B = fp16(p) * s_tg (the group's per-token scale), so
//       O = MMA(codes + 1024, P s) - 1024 MMA(1, P s) + MMA(m, P):
//     the bias and the per-token offsets m are two small MMAs (rows = groups).
// KIVI's newest tokens (its full-precision residual ring) are read from
// global memory as bf16 rows in the same layout.
#include <type_traits>

#include "decode_attn.cuh"
#include "stream_common.cuh"

namespace kvq {
namespace {
using namespace dattn;
using namespace stream;

// blocks per ring stage (copied together): 16 (half the producer's per-stage
// bookkeeping of 8-block stages; 77.9 -> 73.4 us on the 8B-shaped KIVI cache),
// where KVarN's larger blocks keep stream_common's 8
constexpr int kSBD = 16;

template <int D, int KB, int VB, int FMT>
struct SCfg {
  static constexpr int NG = D / 32;                    // groups of 32 channels
  static constexpr int KS_STEPS = D / 16;              // MMA k-steps over channels
  static constexpr int MT = D / 16;                    // P V m-tiles (channels)
  static constexpr bool KIVI = FMT == KVQ_FMT_KIVI;
  static constexpr bool SYM = FMT == KVQ_FMT_SYMMETRIC;
  static constexpr int KCB = D * KB / 8, VCB = D * VB / 8;   // code bytes per token
  // per block: K metadata (KIVI: one row of D per block; else per token), V metadata
  static constexpr int KMETA = KIVI ? D * 2 : kBT * NG * 2;
  static constexpr int VMETA = kBT * NG * 2;
  // a stage holds kSBD consecutive blocks, each plane contiguous over them
  static constexpr int KC = 0;
  static constexpr int VC = KC + kSBD * kBT * KCB;
  static constexpr int KS = VC + kSBD * kBT * VCB;
  static constexpr int KZ = KS + kSBD * KMETA;
  static constexpr int VS = KZ + (SYM ? 0 : kSBD * KMETA);
  static constexpr int VZ = VS + kSBD * VMETA;
  static constexpr int STAGE = (VZ + (SYM ? 0 : kSBD * VMETA) + 127) / 128 * 128;
};

// Two tokens' fp16 metadata of group gq packed as (token a, token b), from
// each token's NG values loaded as 32-bit words.
__device__ __forceinline__ uint32_t pair_group(uint32_t wa, uint32_t wb, int gq) {
  return __byte_perm(wa, wb, (gq & 1) ? 0x7632 : 0x5410);
}

// KIVI keys, read in place.  A 32-bit word of a token's codes holds CPW
// channels, the first CPW / 2 in its low half and the rest in its high half,
// each at bit KB p of its half.  (w >> sh) & (mask << KB j) | 0x64006400 is
// the pair (channel p, channel CPW / 2 + p) as fp16 1024 + c 2^(KB j) for
// p = PER sh / (KB PER) + j, j < PER: a LOP3 per pair (and a shift per PER
// pairs).  PER keeps 2^(KB j) <= 16, so the weights 2^-(KB j) folded into the
// query operand and 2^(KB j) into the zero points stay far from fp16's range.
// Register i of a thread is position i % RPW of its code word i / RPW; the
// thread reads words tid NWT .. tid NWT + NWT - 1 of a token.
template <int D, int KB>
struct KPos {
  static constexpr int CPW = 32 / KB;                 // channels per code word
  static constexpr int RPW = CPW / 2;                 // register pairs per word
  static constexpr int NWT = D * KB / 128;            // code words per thread and token
  static constexpr int NR = NWT * RPW;                // = D / 8 registers per token
  static constexpr int PER = KB == 2 ? 3 : 2;         // positions per shift
  static constexpr uint32_t MASK = KB == 2 ? 0x00030003u : 0x000F000Fu;
  __host__ __device__ static constexpr int e(int p) { return KB * (p % PER); }
  // channels (within the thread's D / 4) of register i's low and high halves
  __host__ __device__ static constexpr int lo(int i) { return (i / RPW) * CPW + i % RPW; }
  __host__ __device__ static constexpr int hi(int i) { return lo(i) + CPW / 2; }
  // register i from its code word w
  __device__ static __forceinline__ uint32_t get(int i, uint32_t w) {
    const int p = i % RPW;
    return magic2h(w >> (KB * PER * (p / PER)), MASK << e(p));
  }
};
// fp16 pair (2^e, 2^e), 0 <= e <= 15
__host__ __device__ constexpr uint32_t pow2_h2(int e) {
  return ((uint32_t)(15 + e) << 10) | ((uint32_t)(15 + e) << 26);
}

template <int D, int KB, int VB, int FMT, bool RAG>
__global__ void __launch_bounds__(kThreads, 1)
decode_stream_kernel(Geom g, const __nv_bfloat16* __restrict__ q, float scale, int* err,
                     __nv_bfloat16* __restrict__ out, int ns) {
  using C = SCfg<D, KB, VB, FMT>;
  constexpr int NG = C::NG, KSS = C::KS_STEPS, MT = C::MT;
  extern __shared__ __align__(128) unsigned char smem[];
  pdl_wait();
  pdl_trigger();

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int gid = lane >> 2, tid = lane & 3;
  const int grp = g.Hq / g.H;
  const int PW = grp * (D + 2);                      // floats of one warp's partial
  float* slot = reinterpret_cast<float*>(smem + (size_t)ns * C::STAGE);   // [kNW][PW]
  Merge* mg = reinterpret_cast<Merge*>(slot + kNW * PW);
  uint64_t* full = reinterpret_cast<uint64_t*>(mg + 1);
  uint64_t* empty = full + ns;
  // ragged / paged caches: each sequence's tokens and first flattened block
  int* s_T = reinterpret_cast<int*>(empty + ns);     // [B]
  int64_t* s_pre = reinterpret_cast<int64_t*>(s_T + ((g.B + 1) & ~1));   // [B + 1]

  // RAG: a ragged or paged cache (a separate instantiation, so the uniform
  // kernel carries none of the per-sequence bookkeeping)
  constexpr bool rag = RAG;
  const bool paged = RAG && g.layout == KVQ_LAYOUT_PAGED;
  const int T = rag ? 0 : cache_tokens(g);
  const int BH = g.B * g.H;
  const int nb = (T + kBT - 1) / kBT;                // blocks per head (uniform layout)
  if (rag) {
    // s_pre[b] = blocks of the sequences before b (H heads each): one warp,
    // 32 sequences per step, a shuffle scan within the step
    if (warp == 0) {
      int64_t run = 0;
      for (int b0 = 0; b0 < g.B; b0 += 32) {
        const int b = b0 + lane;
        const int tb = b < g.B ? *reinterpret_cast<volatile int32_t*>(&g.seq_len[b]) : 0;
        if (b < g.B) s_T[b] = tb;
        int64_t x = (int64_t)g.H * ((tb + kBT - 1) / kBT), incl = x;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int64_t y = __shfl_up_sync(0xffffffffu, incl, o);
          if (lane >= o) incl += y;
        }
        if (b < g.B) s_pre[b] = run + incl - x;
        run += __shfl_sync(0xffffffffu, incl, 31);
      }
      if (lane == 0) s_pre[g.B] = run;
    }
    __syncthreads();
    // a sequence holding no token attends to nothing: zero output (no block
    // of the flattened space belongs to it, so no CTA writes it otherwise)
    if (blockIdx.x == 0)
      for (int i = threadIdx.x; i < g.B * g.Hq * D; i += blockDim.x)
        if (s_T[i / (g.Hq * D)] == 0) out[i] = __float2bfloat16(0.f);
  }
  const int64_t N = rag ? s_pre[g.B] : (int64_t)BH * nb;
  if (N == 0) {                                      // nothing stored: zero output
    if (blockIdx.x == 0 && !rag)
      for (int i = threadIdx.x; i < g.B * g.Hq * D; i += blockDim.x) out[i] = __float2bfloat16(0.f);
    return;
  }
  // head hd = b H + hkv: its tokens, blocks and first flattened block; the
  // head holding flattened block k
  auto T_of = [&](int hd) { return rag ? s_T[hd / g.H] : T; };
  auto nb_of = [&](int hd) { return rag ? (s_T[hd / g.H] + kBT - 1) / kBT : nb; };
  auto start_of = [&](int hd) -> int64_t {
    if (!rag) return (int64_t)hd * nb;
    const int b = hd / g.H;
    return s_pre[b] + (int64_t)(hd - b * g.H) * nb_of(hd);
  };
  auto head_at = [&](int64_t k, int* blk) -> int {
    if (!rag) {
      *blk = (int)(k % nb);
      return (int)(k / nb);
    }
    int lo = 0, hi = g.B - 1;                        // last b with s_pre[b] <= k < s_pre[b + 1]
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (s_pre[mid] <= k) lo = mid; else hi = mid - 1;
    }
    while (s_pre[lo + 1] <= k) ++lo;                 // skip sequences holding no block
    const int nbb = (s_T[lo] + kBT - 1) / kBT;
    const int64_t r = k - s_pre[lo];
    *blk = (int)(r % nbb);
    return lo * g.H + (int)(r / nbb);
  };
  // first byte of head hd's token t in a plane (in a page of a paged cache)
  auto run_ptr = [&](int plane, int hd, int t) -> const uint8_t* {
    int pb = 0, hh = hd;
    int64_t row = t;
    if (paged) {
      tok_loc(g, hd / g.H, t, &pb, &row);
      hh = hd % g.H;
    }
    const Plane& pl = g.pl[plane];
    return static_cast<const uint8_t*>(pl.p) + plane_index(pl, pb, hh, g.H, row, 0) * pl.elem;
  };
  // first byte of head hd's 32-token block k in a per-block plane (KIVI keys)
  auto blk_run_ptr = [&](int plane, int hd, int k) -> const uint8_t* {
    int pb = 0, hh = hd;
    int64_t row = k;
    if (paged) {
      blk_loc(g, hd / g.H, k, &pb, &row);
      hh = hd % g.H;
    }
    const Plane& pl = g.pl[plane];
    return static_cast<const uint8_t*>(pl.p) + plane_index(pl, pb, hh, g.H, row, 0) * pl.elem;
  };
  const int P = N < (int64_t)gridDim.x ? (int)N : (int)gridDim.x;
  if ((int)blockIdx.x >= P) return;
  const int64_t k0 = range_start(blockIdx.x, N, P), k1 = range_start(blockIdx.x + 1, N, P);
  const int nblk = (int)(k1 - k0);
  const int tq = C::KIVI ? kivi_tq(T, g.R, 32) : T;  // coded tokens (uniform layout)
  auto tq_of = [&](int hd) {
    return !rag ? tq : C::KIVI ? kivi_tq(T_of(hd), g.R, 32) : T_of(hd);
  };

  if (threadIdx.x == 0) {
    for (int i = 0; i < ns; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], kSBD);                     // one arrival per block
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncthreads();

  // ------------------------------------------------------------------ producer
  if (warp == kNW) {
    const int nst = (nblk + kSBD - 1) / kSBD;          // stages
    int blk;
    int head = head_at(k0, &blk);                    // first block of the next stage
    // the head's blocks and coded tokens (ragged caches divide to find them)
    int cur_nb = nb_of(head), cur_tq = tq_of(head);
    // bytes of one whole coded block
    constexpr uint32_t kBlockBytes = kBT * (C::KCB + C::VCB) + (C::SYM ? 1 : 2) * kBT * NG * 2 +
                                     (C::KIVI ? 2 * D * 2 : (C::SYM ? 1 : 2) * kBT * NG * 2);
    // copy c (codes of K, V; metadata planes) of a run of r_n blocks of head
    // r_head from its block r_blk into the stage's block slots from r_sub
    auto issue = [&](unsigned char* sp, int st, int myc, int r_head, int r_blk, int r_n,
                     int r_sub) {
      const int t0 = r_blk * kBT;
      const int n4 = (min(r_n * kBT, tq_of(r_head) - t0) + 3) & ~3;
      const int tsub = r_sub * kBT;                  // first token slot in the stage
      const uint8_t* src;
      unsigned char* dst;
      uint32_t bytes;
      if (myc == 0) {
        src = run_ptr(KVQ_PLANE_K_CODES, r_head, t0);
        dst = sp + C::KC + tsub * C::KCB;
        bytes = n4 * C::KCB;
      } else if (myc == 1) {
        src = run_ptr(KVQ_PLANE_V_CODES, r_head, t0);
        dst = sp + C::VC + tsub * C::VCB;
        bytes = n4 * C::VCB;
      } else if (myc == 2 || myc == 4) {
        const int pl = myc == 2 ? KVQ_PLANE_K_SCALE : KVQ_PLANE_K_ZERO;
        src = C::KIVI ? blk_run_ptr(pl, r_head, r_blk) : run_ptr(pl, r_head, t0);
        dst = sp + (myc == 2 ? C::KS : C::KZ) + r_sub * C::KMETA;
        bytes = C::KIVI ? r_n * D * 2 : n4 * NG * 2;
      } else {
        const int pl = myc == 3 ? KVQ_PLANE_V_SCALE : KVQ_PLANE_V_ZERO;
        src = run_ptr(pl, r_head, t0);
        dst = sp + (myc == 3 ? C::VS : C::VZ) + r_sub * C::VMETA;
        bytes = n4 * NG * 2;
      }
      bulk_g2s(dst, src, bytes, &full[st]);
    };
    int s = 0;
    for (; s < nst; ++s) {
      const int st = s % ns;
      bool ok = true;
      if (s >= ns && lane == 0) ok = mbar_wait(&empty[st], ((s / ns) - 1) & 1);
      if (!__shfl_sync(0xffffffffu, ok, 0)) {
        if (lane == 0) atomicOr(err, 1);
        break;
      }
      const int nbs = min(kSBD, nblk - s * kSBD);
      unsigned char* sp = smem + (size_t)st * C::STAGE;
      if (blk + nbs <= cur_nb && (blk + nbs) * kBT <= cur_tq) {
        // the common case: the stage's blocks are whole coded blocks of one
        // head, one run (a paged cache: one run per page it touches, at most 3)
        if (lane == 0) mbar_expect_tx(&full[st], nbs * kBlockBytes);
        __syncwarp();
        constexpr int PB = kPageTok / kBT;               // blocks per page
        const int nsub = paged ? (blk % PB + nbs + PB - 1) / PB : 1;
        const int sub = lane / 6, myc = lane % 6;
        if (sub < nsub && myc < (C::SYM ? 4 : 6)) {
          const int b0 = sub == 0 ? blk : (blk / PB + sub) * PB;
          const int b1 = paged ? min(blk + nbs, (blk / PB + sub + 1) * PB) : blk + nbs;
          issue(sp, st, myc, head, b0, b1 - b0, b0 - blk);
        }
        blk += nbs;
        if (blk == cur_nb) {
          blk = 0;
          ++head;
          while (rag && head < BH && nb_of(head) == 0) ++head;   // sequences holding nothing
          cur_nb = head < BH ? nb_of(head) : 0;
          cur_tq = head < BH ? tq_of(head) : 0;
        }
        continue;
      }
      // split the stage's blocks into runs of one head's coded blocks; in
      // pass p, lane 6 r + c issues copy c of run 5 p + r (every lane walks
      // the same blocks, so the bookkeeping stays in registers)
      const int h_st = head, b_st = blk;             // the stage's first block
      const int nb_st = cur_nb, tq_st = cur_tq;      // and its head's counts
      int nrun = 0;
      uint32_t total = 0;
      for (int pass = 0; pass == 0 || pass * 5 < nrun; ++pass) {
        const int myr = pass * 5 + lane / 6, myc = lane % 6;
        int hh = h_st, bb = b_st, cnt = 0, r_head = 0, r_blk = 0, r_n = 0, r_sub = 0;
        int p_head = -1, p_end = -1;                 // end of the current run
        int nbh = nb_st, tqh = tq_st;                // head hh's blocks and coded tokens
#pragma unroll
        for (int i = 0; i < kSBD; ++i) {
          if (i < nbs && bb * kBT < tqh) {
            // a new run starts here (a paged cache's runs stay in one page)
            if (!(hh == p_head && bb == p_end) || (paged && bb % (kPageTok / kBT) == 0)) {
              if (cnt == myr) { r_head = hh; r_blk = bb; r_sub = i; }
              ++cnt;
            }
            if (cnt - 1 == myr) ++r_n;
            if (pass == 0) {
              // bytes of the block (the last coded block of a head may be
              // partial: whole 4-token groups are copied)
              const int nt = (min(kBT, tqh - bb * kBT) + 3) & ~3;
              total += nt * (C::KCB + C::VCB) + (C::SYM ? 1 : 2) * nt * NG * 2;
              total += C::KIVI ? 2 * D * 2 : (C::SYM ? 1 : 2) * nt * NG * 2;
            }
            p_head = hh;
            p_end = bb + 1;
          }
          if (i < nbs && ++bb == nbh) {
            bb = 0;
            ++hh;
            while (rag && hh < BH && nb_of(hh) == 0) ++hh;   // sequences holding nothing
            nbh = hh < BH ? nb_of(hh) : 0;
            tqh = hh < BH ? tq_of(hh) : 0;
          }
        }
        if (pass == 0) {
          nrun = cnt;
          head = hh;                                 // first block of the next stage
          blk = bb;
          cur_nb = nbh;
          cur_tq = tqh;
          if (lane == 0) mbar_expect_tx(&full[st], total);   // 0: nothing to copy
          __syncwarp();
        }
        if (lane < 30 && myr < nrun && (!C::SYM || myc < 4))
          issue(sp, st, myc, r_head, r_blk, r_n, r_sub);
      }
    }
    // keep the CTA alive until the last copies have landed (the consumers
    // wait for them too, unless they gave up on a timeout)
    if (lane == 0)
      for (int i = max(0, s - ns); i < s; ++i)
        if (!mbar_wait(&full[i % ns], (i / ns) & 1)) atomicOr(err, 1);
    return;
  }

  // ------------------------------------------------------------------ consumers
  const float c2 = scale * 1.4426950408889634f;      // scores in log2 units
  const uint32_t kmask = KB == 4 ? 0x000F000Fu : 0x00030003u;
  const uint32_t vmask = VB == 4 ? 0x000F000Fu : 0x00030003u;
  const int zb = C::SYM ? (1 << (KB - 1)) : 0;       // symmetric key code bias
  const int zbv = C::SYM ? (1 << (VB - 1)) : 0;
  // values: bits between a thread's consecutive channels, and the bit of the
  // channel of row gid in m-tile u (see the P V step)
  constexpr int SH = VB == 4 ? 4 : 2;
  auto vsh = [](int u) { return VB == 4 ? 0 : 2 * SH * u; };
  const int tc = threadIdx.x;                        // 0 .. kNW * 32 - 1
  float* wsb = reinterpret_cast<float*>(g.pl[KVQ_PLANE_WORKSPACE].p);

  int b = 0, hkv = 0;
  bool bad = false;                                  // a wait timed out: stop computing
  using KP = KPos<D, KB>;
  // per-token keys: B fragments of q (head gid) and per-group sums of q;
  // KIVI keys: q of head gid in the positional layout, q_d 2^-e as fp16
  uint32_t qb[C::KIVI ? 1 : KSS][2];
  float qs[C::KIVI ? 1 : NG][2];
  uint32_t qw[C::KIVI ? KP::NR : 1];
  float m_run[2], l_run[2];
  float o[MT][4], bias[NG][4], offa[4];
  bool folded = false;          // the coded blocks' terms are folded into o

  // bf16 B fragments of q in the qk_chan layout (head gid, channels 32 gq + 8 tid + e)
  auto q_frags = [&](uint32_t (&f)[KSS][2]) {
    const __nv_bfloat16* qh = q + ((int64_t)b * g.Hq + hkv * grp) * D;
#pragma unroll
    for (int gq = 0; gq < NG; ++gq) {
      uint4 u = make_uint4(0, 0, 0, 0);
      if (gid < grp) u = *reinterpret_cast<const uint4*>(qh + gid * D + 32 * gq + 8 * tid);
      const uint16_t* e = reinterpret_cast<const uint16_t*>(&u);
#pragma unroll
      for (int sub = 0; sub < 2; ++sub) {
        f[2 * gq + sub][0] = pack_raw(e[qk_chan<KB>(sub, 0, 0)], e[qk_chan<KB>(sub, 0, 1)]);
        f[2 * gq + sub][1] = pack_raw(e[qk_chan<KB>(sub, 1, 0)], e[qk_chan<KB>(sub, 1, 1)]);
      }
    }
  };

  auto load_q = [&]() {
    const __nv_bfloat16* qh = q + ((int64_t)b * g.Hq + hkv * grp) * D;
    if constexpr (C::KIVI) {
      const __nv_bfloat16* qr = qh + gid * D + tid * (D / 4);
#pragma unroll
      for (int i = 0; i < KP::NR; ++i) {
        const float sc = 1.f / (float)(1 << KP::e(i % KP::RPW));
        qw[i] = gid < grp ? pack_f16(__bfloat162float(qr[KP::lo(i)]) * sc,
                                     __bfloat162float(qr[KP::hi(i)]) * sc)
                          : 0u;
      }
    } else {
#pragma unroll
    for (int gq = 0; gq < NG; ++gq) {
      uint4 u = make_uint4(0, 0, 0, 0);
      if (gid < grp) u = *reinterpret_cast<const uint4*>(qh + gid * D + 32 * gq + 8 * tid);
      const uint16_t* e = reinterpret_cast<const uint16_t*>(&u);
#pragma unroll
      for (int sub = 0; sub < 2; ++sub) {
        qb[2 * gq + sub][0] = pack_raw(e[qk_chan<KB>(sub, 0, 0)], e[qk_chan<KB>(sub, 0, 1)]);
        qb[2 * gq + sub][1] = pack_raw(e[qk_chan<KB>(sub, 1, 0)], e[qk_chan<KB>(sub, 1, 1)]);
      }
      const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&u);
      float s = 0.f;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float2 f = __bfloat1622float2(h2[i]);
        s += f.x + f.y;
      }
      s += __shfl_xor_sync(0xffffffffu, s, 1);
      s += __shfl_xor_sync(0xffffffffu, s, 2);       // head gid, group gq
      qs[gq][0] = __shfl_sync(0xffffffffu, s, 4 * (2 * tid));
      qs[gq][1] = __shfl_sync(0xffffffffu, s, 4 * (2 * tid + 1));
    }
    }
    m_run[0] = m_run[1] = -INFINITY;
    l_run[0] = l_run[1] = 0.f;
#pragma unroll
    for (int i = 0; i < MT; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
#pragma unroll
    for (int i = 0; i < NG; ++i) bias[i][0] = bias[i][1] = bias[i][2] = bias[i][3] = 0.f;
    offa[0] = offa[1] = offa[2] = offa[3] = 0.f;
    folded = false;
  };

  // Fold the coded blocks' code bias (bias[gq] = 1024 sum_t p s_tg), channel
  // weights and offset terms into o.  Done once per head: before the first
  // full-precision block (KIVI's newest tokens, whose values enter o as they
  // are), else after the last block.
  auto fold_o = [&]() {
#pragma unroll
    for (int gq = 0; gq < NG; ++gq) {
      const float b0 = bias[gq][0], b1 = bias[gq][1];
      const float f0 = __shfl_sync(0xffffffffu, offa[0], 4 * gq + tid) - (zbv / 1024.f) * b0;
      const float f1 = __shfl_sync(0xffffffffu, offa[1], 4 * gq + tid) - (zbv / 1024.f) * b1;
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const float w0 = 1.f / (float)(1 << vsh(u)), w1 = 1.f / (float)(1 << (vsh(u) + SH));
        o[2 * gq + u][0] = fmaf(o[2 * gq + u][0] - b0, w0, f0);
        o[2 * gq + u][1] = fmaf(o[2 * gq + u][1] - b1, w0, f1);
        o[2 * gq + u][2] = fmaf(o[2 * gq + u][2] - b0, w1, f0);
        o[2 * gq + u][3] = fmaf(o[2 * gq + u][3] - b1, w1, f1);
      }
    }
    folded = true;
  };

  // one 32-token block: scores, online softmax, P V
  // full: all kBT tokens of the block are stored (every block but a head's
  // last), so the per-token validity checks fold away
  auto process = [&](auto full, const unsigned char* sp, int sub_blk, int t0, int nv_in,
                     bool coded) {
    const int nv = decltype(full)::value ? kBT : nv_in;
    const unsigned char* kcp = sp + C::KC + sub_blk * kBT * C::KCB;
    const unsigned char* vcp = sp + C::VC + sub_blk * kBT * C::VCB;
    const unsigned char* ksp = sp + C::KS + sub_blk * C::KMETA;
    const unsigned char* kzp = sp + C::KZ + sub_blk * C::KMETA;
    const unsigned char* vsp = sp + C::VS + sub_blk * C::VMETA;
    const unsigned char* vzp = sp + C::VZ + sub_blk * C::VMETA;
    float S[2][4];
    if constexpr (!C::KIVI) {
      float acc[NG][2][4];
#pragma unroll
      for (int gq = 0; gq < NG; ++gq)
#pragma unroll
        for (int mt = 0; mt < 2; ++mt) acc[gq][mt][0] = acc[gq][mt][1] = acc[gq][mt][2] = acc[gq][mt][3] = 0.f;
#pragma unroll
      for (int mt = 0; mt < 2; ++mt) {
        const unsigned char* r0 = kcp + (16 * mt + gid) * C::KCB;
        const unsigned char* r1 = r0 + 8 * C::KCB;
#pragma unroll
        for (int gq = 0; gq < NG; ++gq) {
          uint32_t w0, w1;
          if (KB == 4) {
            w0 = *reinterpret_cast<const uint32_t*>(r0 + 16 * gq + 4 * tid);
            w1 = *reinterpret_cast<const uint32_t*>(r1 + 16 * gq + 4 * tid);
          } else {
            const uint32_t v0 = *reinterpret_cast<const uint16_t*>(r0 + 8 * gq + 2 * tid);
            const uint32_t v1 = *reinterpret_cast<const uint16_t*>(r1 + 8 * gq + 2 * tid);
            w0 = v0 | (v0 << 14);
            w1 = v1 | (v1 << 14);
          }
#pragma unroll
          for (int sub = 0; sub < 2; ++sub) {
            uint32_t a[4];
            a[0] = magic2(w0 >> (8 * sub), kmask);
            a[1] = magic2(w1 >> (8 * sub), kmask);
            a[2] = magic2(w0 >> (8 * sub + 4), kmask);
            a[3] = magic2(w1 >> (8 * sub + 4), kmask);
            mma16816(acc[gq][mt], a, qb[2 * gq + sub][0], qb[2 * gq + sub][1]);
          }
        }
      }
      const __half* ksc = reinterpret_cast<const __half*>(ksp);
      const __half* kze = reinterpret_cast<const __half*>(kzp);
#pragma unroll
      for (int mt = 0; mt < 2; ++mt)
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          const int t = 16 * mt + gid + 8 * r;
          float s0 = 0.f, s1 = 0.f;
#pragma unroll
          for (int gq = 0; gq < NG; gq += 2) {
            const float2 sc = __half22float2(*reinterpret_cast<const __half2*>(ksc + t * NG + gq));
            float2 mz;
            if (C::SYM) mz = make_float2(-(float)zb * sc.x, -(float)zb * sc.y);
            else mz = __half22float2(*reinterpret_cast<const __half2*>(kze + t * NG + gq));
            const float off0 = mz.x - 128.f * sc.x, off1 = mz.y - 128.f * sc.y;
            s0 += sc.x * acc[gq][mt][2 * r] + off0 * qs[gq][0];
            s1 += sc.x * acc[gq][mt][2 * r + 1] + off0 * qs[gq][1];
            s0 += sc.y * acc[gq + 1][mt][2 * r] + off1 * qs[gq + 1][0];
            s1 += sc.y * acc[gq + 1][mt][2 * r + 1] + off1 * qs[gq + 1][1];
          }
          const bool valid = t < nv;
          S[mt][2 * r] = valid ? s0 * c2 : -INFINITY;
          S[mt][2 * r + 1] = valid ? s1 * c2 : -INFINITY;
        }
    } else if (coded) {
      // KIVI keys (one scale s_d and zero z_d per block and channel):
      //   S_h = sum_d (q_hd s_d) c_d + sum_d q_hd z_d
      // A = codes in place (1024 + c 2^e), B = q 2^-e s as fp16 hi + lo.
      // the block's scales and zeros of the thread's D / 4 channels, as pairs
      const uint32_t* sw = reinterpret_cast<const uint32_t*>(ksp) + tid * (D / 8);
      const uint32_t* zw = reinterpret_cast<const uint32_t*>(kzp) + tid * (D / 8);
      // code words of rows gid, gid + 8 of both 16-token halves
      uint32_t cw[2][2][KP::NWT];
#pragma unroll
      for (int mt = 0; mt < 2; ++mt)
#pragma unroll
        for (int rr = 0; rr < 2; ++rr) {
          const uint32_t* row = reinterpret_cast<const uint32_t*>(
              kcp + (16 * mt + gid + 8 * rr) * C::KCB) + tid * KP::NWT;
#pragma unroll
          for (int m = 0; m < KP::NWT; ++m) cw[mt][rr][m] = row[m];
        }
      // sz rows 0-7: sum_d q s 2^-e, rows 8-15: sum_d q z (heads in the columns)
      float acc[2][4] = {}, sz[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int ks = 0; ks < KSS; ++ks) {
        // B = q 2^-e s split exactly into fp16 hi + lo (an FMA gives the
        // product's rounding error); the scales (A rows 0-7) and the weighted
        // zeros (rows 8-15) against B = q 2^-e give sum_d q s 2^-e and
        // sum_d q z exactly
        uint32_t bh[2], bl[2], as[2], az[2];
#pragma unroll
        for (int hf = 0; hf < 2; ++hf) {
          const int i = 2 * ks + hf;
          const int sel = (KP::lo(i) & 1) ? 0x7632 : 0x5410;
          as[hf] = __byte_perm(sw[KP::lo(i) >> 1], sw[KP::hi(i) >> 1], sel);
          az[hf] = hmul2u(__byte_perm(zw[KP::lo(i) >> 1], zw[KP::hi(i) >> 1], sel),
                          pow2_h2(KP::e(i % KP::RPW)));
          bh[hf] = hmul2u(qw[i], as[hf]);
          bl[hf] = hfma2u_neg(qw[i], as[hf], bh[hf]);
        }
        const uint32_t aSZ[4] = {as[0], az[0], as[1], az[1]};
        mma16816_f16(sz, aSZ, qw[2 * ks], qw[2 * ks + 1]);
#pragma unroll
        for (int mt = 0; mt < 2; ++mt) {
          const int i0 = 2 * ks, i1 = 2 * ks + 1;
          const int m0 = i0 / KP::RPW, m1 = i1 / KP::RPW;
          uint32_t a[4];
          a[0] = KP::get(i0, cw[mt][0][m0]);
          a[1] = KP::get(i0, cw[mt][1][m0]);
          a[2] = KP::get(i1, cw[mt][0][m1]);
          a[3] = KP::get(i1, cw[mt][1][m1]);
          mma16816_f16(acc[mt], a, bh[0], bh[1]);
          mma16816_f16(acc[mt], a, bl[0], bl[1]);
        }
      }
      // per head (columns 2 tid, 2 tid + 1): sum_d q z less the 1024 terms
      const float cs0 = sz[2] - 1024.f * sz[0];
      const float cs1 = sz[3] - 1024.f * sz[1];
#pragma unroll
      for (int mt = 0; mt < 2; ++mt)
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          const bool valid = 16 * mt + gid + 8 * r < nv;
          S[mt][2 * r] = valid ? (acc[mt][2 * r] + cs0) * c2 : -INFINITY;
          S[mt][2 * r + 1] = valid ? (acc[mt][2 * r + 1] + cs1) * c2 : -INFINITY;
        }
    } else {  // full-precision keys (KIVI residual ring), read from global memory
      uint32_t qb[KSS][2];
      q_frags(qb);
#pragma unroll
      for (int mt = 0; mt < 2; ++mt) {
        float acc[4] = {0.f, 0.f, 0.f, 0.f};
        const int ta = t0 + 16 * mt + gid, tb = ta + 8;
        const __nv_bfloat16* ka = plane_ptr<__nv_bfloat16>(g, KVQ_PLANE_K_FULL, b, hkv, ta < t0 + nv ? ta % g.ring : 0);
        const __nv_bfloat16* kb = plane_ptr<__nv_bfloat16>(g, KVQ_PLANE_K_FULL, b, hkv, tb < t0 + nv ? tb % g.ring : 0);
#pragma unroll
        for (int gq = 0; gq < NG; ++gq) {
          const uint4 ua = ta < t0 + nv ? *reinterpret_cast<const uint4*>(ka + 32 * gq + 8 * tid) : make_uint4(0, 0, 0, 0);
          const uint4 ub = tb < t0 + nv ? *reinterpret_cast<const uint4*>(kb + 32 * gq + 8 * tid) : make_uint4(0, 0, 0, 0);
          const uint16_t* ea = reinterpret_cast<const uint16_t*>(&ua);
          const uint16_t* eb = reinterpret_cast<const uint16_t*>(&ub);
#pragma unroll
          for (int sub = 0; sub < 2; ++sub) {
            uint32_t a[4];
            a[0] = pack_raw(ea[qk_chan<KB>(sub, 0, 0)], ea[qk_chan<KB>(sub, 0, 1)]);
            a[1] = pack_raw(eb[qk_chan<KB>(sub, 0, 0)], eb[qk_chan<KB>(sub, 0, 1)]);
            a[2] = pack_raw(ea[qk_chan<KB>(sub, 1, 0)], ea[qk_chan<KB>(sub, 1, 1)]);
            a[3] = pack_raw(eb[qk_chan<KB>(sub, 1, 0)], eb[qk_chan<KB>(sub, 1, 1)]);
            mma16816(acc, a, qb[2 * gq + sub][0], qb[2 * gq + sub][1]);
          }
        }
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          const bool valid = 16 * mt + gid + 8 * r < nv;
          S[mt][2 * r] = valid ? acc[2 * r] * c2 : -INFINITY;
          S[mt][2 * r + 1] = valid ? acc[2 * r + 1] * c2 : -INFINITY;
        }
      }
    }

    // --------------------------------------------------------------- softmax
    float mx[2];
#pragma unroll
    for (int jh = 0; jh < 2; ++jh) {
      mx[jh] = fmaxf(fmaxf(S[0][jh], S[0][2 + jh]), fmaxf(S[1][jh], S[1][2 + jh]));
      mx[jh] = fmaxf(mx[jh], __shfl_xor_sync(0xffffffffu, mx[jh], 4));
      mx[jh] = fmaxf(mx[jh], __shfl_xor_sync(0xffffffffu, mx[jh], 8));
      mx[jh] = fmaxf(mx[jh], __shfl_xor_sync(0xffffffffu, mx[jh], 16));
    }
    float alpha[2];
#pragma unroll
    for (int jh = 0; jh < 2; ++jh) {
      const float mn = fmaxf(m_run[jh], mx[jh]);
      alpha[jh] = m_run[jh] == -INFINITY ? 0.f : exp2f(m_run[jh] - mn);
      m_run[jh] = mn;
      l_run[jh] *= alpha[jh];
    }
    if (__any_sync(0xffffffffu, alpha[0] != 1.f || alpha[1] != 1.f)) {
#pragma unroll
      for (int i = 0; i < MT; ++i) {
        o[i][0] *= alpha[0]; o[i][1] *= alpha[1];
        o[i][2] *= alpha[0]; o[i][3] *= alpha[1];
      }
#pragma unroll
      for (int i = 0; i < NG; ++i) {
        bias[i][0] *= alpha[0]; bias[i][1] *= alpha[1];
        bias[i][2] *= alpha[0]; bias[i][3] *= alpha[1];
      }
      offa[0] *= alpha[0]; offa[1] *= alpha[1];
      offa[2] *= alpha[0]; offa[3] *= alpha[1];
    }
    uint32_t pb[2][2];                               // B fragments of P^T per 16-token step
#pragma unroll
    for (int mt = 0; mt < 2; ++mt) {
      float p[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        p[i] = exp2f(S[mt][i] - m_run[i & 1]);       // exp2(-inf) = 0
        l_run[i & 1] += p[i];
      }
      pb[mt][0] = movmatrix_t(pack_f16(p[0], p[1]));
      pb[mt][1] = movmatrix_t(pack_f16(p[2], p[3]));
    }

    // ------------------------------------------------------------------- P V
    if (coded) {
#pragma unroll
      for (int mt = 0; mt < 2; ++mt) {
        int tk[4];
        uint32_t vsw[4][(NG + 1) / 2];               // per token: NG fp16 scales as words
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          tk[i] = 16 * mt + 2 * tid + (i & 1) + 8 * (i >> 1);
          const bool v = tk[i] < nv;
          const uint32_t* src = reinterpret_cast<const uint32_t*>(vsp + tk[i] * NG * 2);
#pragma unroll
          for (int w = 0; w < (NG + 1) / 2; ++w) vsw[i][w] = v ? src[w] : 0u;
        }
        if (!C::SYM) {                               // offsets: rows = groups
          uint32_t a[4] = {0u, 0u, 0u, 0u};
          if (gid < NG) {
            const uint16_t* vz = reinterpret_cast<const uint16_t*>(vzp);
            uint32_t z[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) z[i] = tk[i] < nv ? vz[tk[i] * NG + gid] : 0u;
            a[0] = z[0] | (z[1] << 16);
            a[2] = z[2] | (z[3] << 16);
          }
          mma16816_f16(offa, a, pb[mt][0], pb[mt][1]);
        }
#pragma unroll
        for (int gq = 0; gq < NG; ++gq) {
          const uint32_t s01 = pair_group(vsw[0][gq >> 1], vsw[1][gq >> 1], gq);
          const uint32_t s89 = pair_group(vsw[2][gq >> 1], vsw[3][gq >> 1], gq);
          const uint32_t b0 = hmul2u(pb[mt][0], s01), b1 = hmul2u(pb[mt][1], s89);
          const unsigned char* vc = vcp;
          uint32_t x01, x89;
          if (VB == 4) {
            x01 = (uint32_t)*reinterpret_cast<const uint16_t*>(vc + tk[0] * C::VCB + 16 * gq + 2 * gid) |
                  ((uint32_t)*reinterpret_cast<const uint16_t*>(vc + tk[1] * C::VCB + 16 * gq + 2 * gid) << 16);
            x89 = (uint32_t)*reinterpret_cast<const uint16_t*>(vc + tk[2] * C::VCB + 16 * gq + 2 * gid) |
                  ((uint32_t)*reinterpret_cast<const uint16_t*>(vc + tk[3] * C::VCB + 16 * gq + 2 * gid) << 16);
          } else {
            x01 = (uint32_t)vc[tk[0] * C::VCB + 8 * gq + gid] | ((uint32_t)vc[tk[1] * C::VCB + 8 * gq + gid] << 16);
            x89 = (uint32_t)vc[tk[2] * C::VCB + 8 * gq + gid] | ((uint32_t)vc[tk[3] * C::VCB + 8 * gq + gid] << 16);
          }
          // rows gid and gid + 8 of m-tile u are the channels at bits vsh(u)
          // and vsh(u) + SH of each half, read in place as 1024 + c 2^bit
          // (4-bit: the upper pair after a shift by 8); the weights come
          // off when the head's output is folded
#pragma unroll
          for (int u = 0; u < 2; ++u) {
            const uint32_t y01 = (VB == 4 && u) ? x01 >> 8 : x01;
            const uint32_t y89 = (VB == 4 && u) ? x89 >> 8 : x89;
            uint32_t a[4];
            a[0] = magic2h(y01, vmask << vsh(u));
            a[1] = magic2h(y01, vmask << (vsh(u) + SH));
            a[2] = magic2h(y89, vmask << vsh(u));
            a[3] = magic2h(y89, vmask << (vsh(u) + SH));
            mma16816_f16(o[2 * gq + u], a, b0, b1);
          }
          const uint32_t ab[4] = {kMagicH, kMagicH, kMagicH, kMagicH};
          mma16816_f16(bias[gq], ab, b0, b1);
        }
      }
    } else {  // full-precision values
      if (!folded) fold_o();
#pragma unroll
      for (int mt = 0; mt < 2; ++mt) {
        const __nv_bfloat16* vr[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int t = t0 + 16 * mt + 2 * tid + (i & 1) + 8 * (i >> 1);
          vr[i] = t < t0 + nv ? plane_ptr<__nv_bfloat16>(g, KVQ_PLANE_V_FULL, b, hkv, t % g.ring) : nullptr;
        }
#pragma unroll
        for (int gq = 0; gq < NG; ++gq) {
          uint2 vw[4];
#pragma unroll
          for (int i = 0; i < 4; ++i)
            vw[i] = vr[i] ? *reinterpret_cast<const uint2*>(vr[i] + 32 * gq + 4 * gid) : make_uint2(0, 0);
          auto el = [&](int i, int c) {
            const __nv_bfloat16* e = reinterpret_cast<const __nv_bfloat16*>(&vw[i]);
            return __bfloat162float(e[c]);
          };
#pragma unroll
          for (int u = 0; u < 2; ++u) {
            uint32_t a[4];
            a[0] = pack_f16(el(0, 2 * u), el(1, 2 * u));
            a[1] = pack_f16(el(0, 2 * u + 1), el(1, 2 * u + 1));
            a[2] = pack_f16(el(2, 2 * u), el(3, 2 * u));
            a[3] = pack_f16(el(2, 2 * u + 1), el(3, 2 * u + 1));
            mma16816_f16(o[2 * gq + u], a, pb[mt][0], pb[mt][1]);
          }
        }
      }
    }
  };

  // ------------------------------------------------------ head segments
  // The CTA's range crosses heads hfirst..hlast.  Every consumer warp runs
  // every segment (warps without blocks in it only join the merge), so the
  // named barriers below are reached by all of them.
  int bdummy;
  const int hfirst = head_at(k0, &bdummy), hlast = head_at(k1 - 1, &bdummy);
  for (int hd = hfirst; hd <= hlast; ++hd) {
    const int nbh = nb_of(hd);
    if (nbh == 0) continue;                          // a sequence holding no token
    const int64_t hs = start_of(hd);
    const int a = (int)(max(k0, hs) - k0), e = (int)(min(k1, hs + nbh) - k0);
    const int Th = T_of(hd), tqh = tq_of(hd);
    b = hd / g.H;
    hkv = hd % g.H;
    const int jst = a + ((warp - a) % kNW + kNW) % kNW;   // first block of this warp
    const bool mine = jst < e;
    if (mine) load_q();
    for (int j = jst; j < e && !bad; j += kNW) {
      const int sj = j / kSBD, st = sj % ns;
      bool ok = true;
      if (lane == 0) ok = mbar_wait(&full[st], (sj / ns) & 1);
      if (!__shfl_sync(0xffffffffu, ok, 0)) {
        if (lane == 0) atomicOr(err, 1);
        bad = true;
        break;
      }
      const int t0 = (int)(k0 + j - hs) * kBT;
      const int nv = min(kBT, Th - t0);
      if (nv == kBT)
        process(std::true_type(), smem + (size_t)st * C::STAGE, j % kSBD, t0, nv, t0 < tqh);
      else
        process(std::false_type(), smem + (size_t)st * C::STAGE, j % kSBD, t0, nv, t0 < tqh);
      __syncwarp();
      if (lane == 0) mbar_arrive1(&empty[st]);
    }
    if (mine) {
      if (!folded) fold_o();
      // reduce l over the rows
#pragma unroll
      for (int jh = 0; jh < 2; ++jh) {
        l_run[jh] += __shfl_xor_sync(0xffffffffu, l_run[jh], 4);
        l_run[jh] += __shfl_xor_sync(0xffffffffu, l_run[jh], 8);
        l_run[jh] += __shfl_xor_sync(0xffffffffu, l_run[jh], 16);
        if (bad) m_run[jh] = -INFINITY;
      }
    }
    consumer_sync();                                 // the previous merge is done with the slots
    if (mine) {
      float* ws = slot + warp * PW;
#pragma unroll
      for (int i = 0; i < MT; ++i) {
        const int d0 = 32 * (i >> 1) + 4 * gid + 2 * (i & 1);
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          const int h = 2 * tid + (r & 1);
          if (h < grp) ws[h * (D + 2) + 2 + d0 + (r >> 1)] = o[i][r];
        }
      }
      if (gid == 0)
#pragma unroll
        for (int jh = 0; jh < 2; ++jh)
          if (2 * tid + jh < grp) {
            ws[(2 * tid + jh) * (D + 2)] = m_run[jh];
            ws[(2 * tid + jh) * (D + 2) + 1] = l_run[jh];
          }
    }
    consumer_sync();
    // merge the warps' partials: warps (a + i) % kNW, i < np, hold this head
    const int np = min(kNW, e - a);
    if (tc < grp) {
      float M = -INFINITY;
      for (int i = 0; i < np; ++i) M = fmaxf(M, slot[((a + i) % kNW) * PW + tc * (D + 2)]);
      float L = 0.f;
      for (int i = 0; i < np; ++i) {
        const float* pp = slot + ((a + i) % kNW) * PW + tc * (D + 2);
        const float w = pp[0] == -INFINITY ? 0.f : exp2f(pp[0] - M);
        mg->m[i][tc] = w;
        L += w * pp[1];
      }
      mg->M[tc] = M;
      mg->L[tc] = L;
    }
    consumer_sync();
    const int c0 = cta_of(hs, N, P), c1 = cta_of(hs + nbh - 1, N, P);
    const int nct = c1 - c0 + 1;
    if (nct > kMaxSplits) {                          // the host sizes the grid so this cannot happen
      if (tc == 0) atomicOr(err, 4);
      continue;
    }
    const int64_t orow0 = (int64_t)b * g.Hq + hkv * grp;
    for (int idx = tc; idx < grp * D; idx += kNW * 32) {
      const int h = idx / D, d = idx % D;
      float acc = 0.f;
      for (int i = 0; i < np; ++i) acc += mg->m[i][h] * slot[((a + i) % kNW) * PW + h * (D + 2) + 2 + d];
      if (nct == 1) {
        const float L = mg->L[h];
        out[(orow0 + h) * D + d] = __float2bfloat16(L > 0.f ? acc / L : 0.f);
      } else {
        wsb[((orow0 + h) * kMaxSplits + (blockIdx.x - c0)) * (D + kWsStride) + 2 + d] = acc;
      }
    }
    if (nct == 1) continue;
    if (tc < grp) {
      float* wr = wsb + ((orow0 + tc) * kMaxSplits + (blockIdx.x - c0)) * (D + kWsStride);
      wr[0] = mg->M[tc];
      wr[1] = mg->L[tc];
    }
    // the last CTA of this head merges all of its CTAs' partials
    consumer_sync();
    if (tc == 0) {
      __threadfence();
      mg->last = atomicAdd(&g.counters[hd], 1u) == (unsigned)nct - 1;
    }
    consumer_sync();
    if (!mg->last) continue;
    __threadfence();
    if (tc < grp * nct) {
      const int h = tc / nct, i = tc % nct;
      const float* wr = wsb + ((orow0 + h) * kMaxSplits + i) * (D + kWsStride);
      mg->m[i][h] = __ldcg(wr);
      mg->l[i][h] = __ldcg(wr + 1);
    }
    consumer_sync();
    if (tc < grp) {
      float M = -INFINITY;
      for (int i = 0; i < nct; ++i) M = fmaxf(M, mg->m[i][tc]);
      float L = 0.f;
      for (int i = 0; i < nct; ++i) {
        const float w = mg->m[i][tc] == -INFINITY ? 0.f : exp2f(mg->m[i][tc] - M);
        mg->m[i][tc] = w;
        L += w * mg->l[i][tc];
      }
      mg->L[tc] = L;
    }
    consumer_sync();
    for (int idx = tc; idx < grp * D; idx += kNW * 32) {
      const int h = idx / D, d = idx % D;
      const float* wr = wsb + (orow0 + h) * kMaxSplits * (D + kWsStride) + 2 + d;
      float acc = 0.f;
#pragma unroll 4
      for (int i = 0; i < nct; ++i) acc += mg->m[i][h] * __ldcg(wr + i * (D + kWsStride));
      const float L = mg->L[h];
      out[(orow0 + h) * D + d] = __float2bfloat16(L > 0.f ? acc / L : 0.f);
    }
    if (tc == 0) g.counters[hd] = 0;                 // ready for the next call
  }
}

template <int D, int KB, int VB, int FMT>
size_t stream_smem(int grp, int B, bool rag, int* ns) {
  using C = SCfg<D, KB, VB, FMT>;
  // per-warp partial slots, merge scratch; ragged: each sequence's count and
  // first block (rounded up so the mbarriers stay 8-byte aligned)
  const size_t fixed = (size_t)kNW * grp * (D + 2) * 4 + sizeof(Merge) +
                       (rag ? (size_t)((B + 2) & ~1) * 4 + (size_t)(B + 1) * 8 : 0);
  int n = (int)((kSmemMax - fixed) / (C::STAGE + 16));
  if (n > kMaxStages) n = kMaxStages;
  *ns = n;
  return (size_t)n * C::STAGE + fixed + (size_t)2 * n * 8;
}

template <int D, int KB, int VB, int FMT>
cudaError_t launch_t(const Geom& g, const void* q, float scale, int* err, void* out,
                     cudaStream_t s) {
  const int grp = g.Hq / g.H;
  int ns = 0;
  const size_t sm = stream_smem<D, KB, VB, FMT>(grp, g.B, g.layout != KVQ_LAYOUT_UNIFORM, &ns);
  auto kern = g.layout == KVQ_LAYOUT_UNIFORM ? decode_stream_kernel<D, KB, VB, FMT, false>
                                             : decode_stream_kernel<D, KB, VB, FMT, true>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
  if (e != cudaSuccess) return e;
  launch_pdl(kern, dim3(decode_stream_ctas(g)), dim3(kThreads), sm, s, g,
             reinterpret_cast<const __nv_bfloat16*>(q), scale, err,
             reinterpret_cast<__nv_bfloat16*>(out), ns);
  return cudaGetLastError();
}

template <int D, int BITS>
cudaError_t launch_fmt(const Geom& g, const void* q, float scale, int* err, void* out,
                       cudaStream_t s) {
  switch (g.fmt) {
    case KVQ_FMT_AFFINE: return launch_t<D, BITS, BITS, KVQ_FMT_AFFINE>(g, q, scale, err, out, s);
    case KVQ_FMT_SYMMETRIC: return launch_t<D, BITS, BITS, KVQ_FMT_SYMMETRIC>(g, q, scale, err, out, s);
    case KVQ_FMT_KIVI: return launch_t<D, BITS, BITS, KVQ_FMT_KIVI>(g, q, scale, err, out, s);
  }
  return cudaErrorNotSupported;
}

}  // namespace

// CTAs of the streaming decode: one per SM, at most 15 per (sequence, kv head)
// so that a head never spans more CTAs than its kMaxSplits workspace rows.
int decode_stream_ctas(const Geom& g) {
  const int bh = g.B * g.H;
  int p = num_sms();
  if (p > 15 * bh) p = 15 * bh;
  // ragged: the longest sequence's heads must not span more CTAs either
  if (g.layout != KVQ_LAYOUT_UNIFORM && g.ragged_cta_cap > 0 && p > g.ragged_cta_cap)
    p = g.ragged_cta_cap;
  return p < 1 ? 1 : p;
}

bool decode_stream_supported(const Geom& g) {
  const bool fmt_ok = g.fmt == KVQ_FMT_AFFINE || g.fmt == KVQ_FMT_SYMMETRIC || g.fmt == KVQ_FMT_KIVI;
  return fmt_ok && g.act == KVQ_BF16 && g.G == 32 && g.kb == g.vb && (g.kb == 2 || g.kb == 4) &&
         (g.D == 64 || g.D == 128) && g.Hq / g.H <= 8;
}

cudaError_t launch_decode_stream(const Geom& g, const void* q, float scale, int* err, void* out,
                                 cudaStream_t s) {
  if (g.D == 64) return g.kb == 4 ? launch_fmt<64, 4>(g, q, scale, err, out, s)
                                  : launch_fmt<64, 2>(g, q, scale, err, out, s);
  return g.kb == 4 ? launch_fmt<128, 4>(g, q, scale, err, out, s)
                   : launch_fmt<128, 2>(g, q, scale, err, out, s);
}

}  // namespace kvq
