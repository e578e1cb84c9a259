// Internal declarations shared by the kvq translation units: the cache
// geometry passed to kernels by value, plane addressing, small device helpers
// and the host-side launch entry points of each kernel family.
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>

#include <utility>
#include <vector>

#include "../../include/kvq.h"

namespace kvq {

constexpr int kMaxSplits = 32;       // decode split-K partials per (b, q head)
constexpr int kWsStride = 2;         // workspace row: m, l, then D outputs

// One plane of the cache: [B][Hkv][rows][cols] elements of `elem` bytes.
struct Plane {
  void* p;
  int64_t rows, cols;
  int32_t elem;
};

// Device-resident state of a cache (first 256 bytes of its buffer).
// tokens: T, the number of stored tokens per sequence; kernels read it, so
// launches do not bake it in and a captured decode step can be replayed.
// done: arrival counter of the last kernel of an append (the last CTA to
// arrive advances `tokens`).  error: bit flags set by kernels that refuse
// work (see kErr*).
struct CacheState {
  int32_t tokens;
  uint32_t done;
  int32_t error;
  int32_t pad[61];
};
constexpr int kErrCapacity = 1;   // an append would exceed max_tokens

// Everything a kernel needs to address a cache.  Passed by value.
struct Geom {
  int32_t fmt, kb, vb, G, R, S, iters;
  int32_t B, H, Hq, D, Tmax, act;
  int32_t ring;          // KIVI: R + G residual slots
  int32_t splits;        // decode split-K width (fixed per cache)
  CacheState* state;
  uint32_t* counters;    // [B][Hkv] split arrival counters (zeroed with the state)
  uint32_t* epoch;       // launch counter of the fused decode step; kept across resets
  Plane pl[KVQ_NUM_PLANES];
  // token layout (kvq_layout).  RAGGED / PAGED: seq_len[b] tokens of sequence
  // b, seq_new[b] of them appended by the last append; PAGED: token t of
  // sequence b in pool page page_table[b max_pages + t / kPageTok], and the
  // planes hold the pool ([1][H][num_pages kPageTok][cols]) instead of
  // [B][H][Tmax][cols]
  int32_t layout, max_pages;
  // RAGGED / PAGED, host side: most streaming-decode CTAs for which no head
  // spans more than kMaxSplits of them at the current lengths (set before
  // each decode launch; 0 = no bound)
  int32_t ragged_cta_cap;
  int32_t* seq_len;
  int32_t* seq_new;
  int32_t* page_table;
};
constexpr int kPageTok = KVQ_PAGE_TOKENS;
constexpr int kPageShift = 8;
static_assert(kPageTok == 1 << kPageShift && kPageTok % 64 == 0,
              "pages hold whole 64-token tiles and decode chunks");

__host__ __device__ inline int64_t plane_index(const Plane& pl, int b, int h, int H,
                                               int64_t row, int64_t col) {
  return (((int64_t)b * H + h) * pl.rows + row) * pl.cols + col;
}

template <typename T>
__host__ __device__ inline T* plane_ptr(const Geom& g, int which, int b, int h,
                                        int64_t row, int64_t col = 0) {
  const Plane& pl = g.pl[which];
  return reinterpret_cast<T*>(pl.p) + plane_index(pl, b, h, g.H, row, col);
}

// KIVI: tokens held as codes once T tokens are stored (whole G-blocks,
// leaving between R and R + G - 1 newest tokens at full precision).
__host__ __device__ inline int kivi_tq(int T, int R, int G) {
  int n = T - R;
  return n > 0 ? (n / G) * G : 0;
}
// KVarN: complete quantized blocks after the sinks.
__host__ __device__ inline int kvarn_nblocks(int T, int S, int G) {
  int n = T - S;
  return n > 0 ? n / G : 0;
}

// Activation loads/stores.
__device__ __forceinline__ float ld_act(const void* p, int64_t i, int act) {
  if (act == KVQ_BF16) return __bfloat162float(reinterpret_cast<const __nv_bfloat16*>(p)[i]);
  return reinterpret_cast<const float*>(p)[i];
}
__device__ __forceinline__ void st_act(void* p, int64_t i, float v, int act) {
  if (act == KVQ_BF16) reinterpret_cast<__nv_bfloat16*>(p)[i] = __float2bfloat16_rn(v);
  else reinterpret_cast<float*>(p)[i] = v;
}

// Programmatic dependent launch: every kernel of the library is launched with
// programmatic stream serialization, so the next grid can be resident while
// the previous one drains.  pdl_wait() (first statement of every kernel)
// blocks until the preceding grid has completed and its memory is visible;
// pdl_trigger() lets the next grid start launching.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t s, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
}

// Host-side launchers (each defined in the translation unit of its kernels).
// They return cudaGetLastError() of their launches.
// All launchers read the token count from g.state on the device.
cudaError_t launch_append(const Geom& g, int L, const void* k, const void* v, cudaStream_t s);
// RAGGED / PAGED: sequence b appends its first n[b] (host array) of L tokens;
// then its device count advances.  seq_reset: sequence b becomes empty.
cudaError_t launch_append_ragged(const Geom& g, int L, const void* k, const void* v,
                                 const int* n, cudaStream_t s);
cudaError_t launch_seq_reset(const Geom& g, int b, cudaStream_t s);
// t_hint: the host's count of stored tokens, used only to choose between
// decode kernels (the kernels read the count from the device).
cudaError_t launch_attend(const Geom& g, const void* q, int L, float scale, void* out,
                          bool decode, int t_hint, cudaStream_t s);
// pos_dev: if non-NULL, positions start at *pos_dev + pos0 (a cache's token
// count read on the device), else at pos0.
cudaError_t launch_project(const void* x, int B, int L, int d_in, const void* w,
                           const void* const a[3], const void* const bm[3], const int r[3],
                           float alpha_over_r, int Hq, int Hkv, int D, int pos0,
                           const int* pos_dev, float rope_base, int act,
                           void* const out[3], int* err, cudaStream_t s, int pos_stride = 0);

// tcgen05 projection (project_tc.cu) for bf16 and more than 16 rows;
// cudaErrorNotSupported if the head shapes do not tile.
// append_to: if non-NULL, k and v are not stored but coded into that cache
// (affine or symmetric, G = 32) at its device token count, which the last CTA
// then advances by B's L tokens (the fused projection-and-append).
cudaError_t launch_project_tc(const void* x, int B, int L, int d_in, const void* w,
                              const void* const a[3], const void* const bm[3], const int r[3],
                              float alpha_over_r, int Hq, int Hkv, int D, int pos0,
                              const int* pos_dev, float rope_base, void* const out[3], int* err,
                              cudaStream_t s, const Geom* append_to = nullptr, int pos_stride = 0);
int project_tc_tile(int Hq, int Hkv, int D, int d_in);
// The same kernel as a plain product: C [M][N] fp32 = A [M][K] B^T, A and Bt
// bf16 K-major, Bt's rows of Kb elements repeated along K (K a multiple of Kb).
cudaError_t launch_gemm_tc_bf16(const void* a, int M, int K, const void* bt, int N, int Kb,
                                float* c, int* err, cudaStream_t s);
// The same kernel over an NF4 base (codes [N][d_in/2], fp32 absmax [N][d_in/64],
// dequantised in the kernel's operand path).
bool project_tc_nf4_supported(int Hq, int Hkv, int D, int d_in);
cudaError_t launch_project_tc_nf4(const void* x, int B, int L, int d_in, const void* codes,
                                  const void* absmax, const void* const a[3],
                                  const void* const bm[3], const int r[3], float alpha_over_r,
                                  int Hq, int Hkv, int D, int pos0, const int* pos_dev,
                                  float rope_base, void* const out[3], int* err, cudaStream_t s,
                                  int pos_stride = 0);

// Projection over an NF4 base (project_nf4.cu): codes [N][d_in/2], fp32 absmax
// [N][d_in/64]; bf16 activations.
bool project_nf4_supported(int d_in, int Hq, int Hkv, int D, const int r[3]);
cudaError_t launch_project_nf4(const void* x, int B, int L, int d_in, const void* codes,
                               const void* absmax, const void* const a[3],
                               const void* const bm[3], const int r[3], float alpha_over_r,
                               int Hq, int Hkv, int D, int pos0, const int* pos_dev,
                               float rope_base, void* const out[3], cudaStream_t s,
                               int pos_stride = 0);
void rope_theta_table(float rope_base, int D, float* hi, float* lo);

// Straight-through backward (backward.cu): attention over a cache's
// reconstruction, then the adapters.  Workspace bytes per (sequence, kv head)
// pair of the attention backward, and of the adapter backward.
size_t attend_backward_pair_bytes(const Geom& g, int T, int L);
cudaError_t launch_attend_backward(const Geom& g, int T, const void* q, const void* d_out,
                                   int L, float scale, float* dq, float* dk, float* dv,
                                   void* ws, size_t ws_bytes, cudaStream_t s);
size_t lora_backward_bytes(int B, int L, int d_in, int Hq, int Hkv, int D, const int r[3]);
cudaError_t launch_lora_backward(const void* x, int B, int L, int d_in, const void* w,
                                 const void* const a[3], const void* const bm[3],
                                 const int r[3], float alpha_over_r, int Hq, int Hkv, int D,
                                 int pos0, float rope_base, int act, const float* dq,
                                 const float* dk, const float* dv, int kv_rows,
                                 float* const da[3], float* const db[3], float* dx, void* ws,
                                 cudaStream_t s);

// Fused decode step (decode_step.cu): projection of the new token, append,
// decode attention in one cooperative kernel.
bool decode_step_supported(const Geom& g, int d_in, const int r[3]);
cudaError_t launch_decode_step(const Geom& g, const void* x, int d_in, const void* w,
                               const void* const a[3], const void* const bm[3], const int r[3],
                               float alpha_over_r, float rope_base, float scale,
                               void* const qkv[3], void* out, int* err, cudaStream_t s);

// Decode split-K width for a cache geometry (fixed, independent of T).
int decode_splits(const Geom& g);

// Tensor-core split decode (attend_mma.cu): the formats it covers, and the
// launch (partials to the workspace plane; the caller merges them).
bool decode_mma_supported(const Geom& g);
// tcgen05 causal prefill with 256 query rows per CTA (attend_prefill_m256.cu).
bool prefill_m256_supported(const Geom& g);
cudaError_t launch_prefill_m256(const Geom& g, const void* q, int L, float scale, void* out,
                                int* err, cudaStream_t s);
// mma.sync causal prefill for the other formats and head dimensions
// (attend_prefill_mma.cu).
bool prefill_mma_supported(const Geom& g);
cudaError_t launch_prefill_mma(const Geom& g, const void* q, int L, float scale, void* out,
                               cudaStream_t s);
cudaError_t launch_decode_mma(const Geom& g, const void* q, float scale, int* err, void* out,
                              cudaStream_t s);
// Streaming persistent decode (decode_stream.cu): the formats it covers, its
// grid size, and the launch (it merges its own partials).
bool decode_stream_supported(const Geom& g);
int decode_stream_ctas(const Geom& g);
cudaError_t launch_decode_stream(const Geom& g, const void* q, float scale, int* err, void* out,
                                 cudaStream_t s);
// Streaming KVarN decode over the coded tokens (decode_stream_kvarn.cu): it
// leaves each head's partial in workspace slot kMaxSplits - 1 for the combine.
bool decode_stream_kvarn_supported(const Geom& g);
cudaError_t launch_decode_stream_kvarn(const Geom& g, const void* q, float scale, int* err,
                                       cudaStream_t s);

// Token range of split `s` of `splits` over T tokens (tiles of `tile`).
__host__ __device__ inline void split_range(int T, int splits, int s, int tile, int* ts,
                                            int* te) {
  int per = (T + splits - 1) / splits;
  per = (per + tile - 1) / tile * tile;
  *ts = s * per;
  *te = min(T, *ts + per);
}

// Token count at the start of an append of L tokens; sets the capacity
// error bit (and the kernels skip all work) if the append would overflow.
__device__ __forceinline__ int append_begin(const Geom& g, int L, bool* ok) {
  const int T0 = *reinterpret_cast<volatile int32_t*>(&g.state->tokens);
  *ok = T0 >= 0 && (int64_t)T0 + L <= g.Tmax;
  if (!*ok && threadIdx.x == 0 && blockIdx.x == 0 && blockIdx.y == 0 && blockIdx.z == 0)
    atomicOr(&g.state->error, kErrCapacity);
  return T0;
}

// Called by every CTA of the final kernel of an append after it has read the
// token count: the last CTA to arrive advances it by L (unless the append
// was refused).
__device__ __forceinline__ void append_arrive(CacheState* st, int T0, int L, bool ok) {
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    const unsigned total = gridDim.x * gridDim.y * gridDim.z;
    const unsigned prev = atomicAdd(&st->done, 1u);
    if (prev == total - 1) {
      if (ok) st->tokens = T0 + L;
      st->done = 0;
      __threadfence();
    }
  }
}

// Batch extent of plane `which`: a paged cache's per-token and per-block
// planes hold the page pool (1); KIVI's full-precision ring stays per sequence.
__host__ __device__ inline int plane_batch(const Geom& g, int which) {
  const bool per_seq = which == KVQ_PLANE_K_FULL || which == KVQ_PLANE_V_FULL ||
                       which == KVQ_PLANE_WORKSPACE;
  return g.layout == KVQ_LAYOUT_PAGED && !per_seq ? 1 : g.B;
}
// Token count before this append, and tokens appended, for sequence b of an
// append of L tokens: the uniform count T0u and L, or a ragged cache's
// seq_len[b] and seq_new[b] (set for this append before its kernels run).
__device__ __forceinline__ void append_span(const Geom& g, int b, int L, int T0u, int* T0,
                                            int* n) {
  if (g.layout == KVQ_LAYOUT_UNIFORM) {
    *T0 = T0u;
    *n = L;
  } else {
    *T0 = g.seq_len[b];
    *n = g.seq_new[b];
  }
}

// Tokens stored, as read by attention kernels.
__device__ __forceinline__ int cache_tokens(const Geom& g) {
  return *reinterpret_cast<volatile int32_t*>(&g.state->tokens);
}
// RoPE position offset of sequence b: *pos_dev for every sequence
// (stride 0), or pos_dev[b] (stride 1: a ragged cache's counts), or 0.
__device__ __forceinline__ int pos_of(const int* pos_dev, int stride, int b) {
  return pos_dev ? pos_dev[b * stride] : 0;
}
// Tokens of sequence b (every layout).
__device__ __forceinline__ int seq_tokens(const Geom& g, int b) {
  return g.layout == KVQ_LAYOUT_UNIFORM ? cache_tokens(g)
                                        : *reinterpret_cast<volatile int32_t*>(&g.seq_len[b]);
}
// Where token t of sequence b sits in a per-token plane: its batch index and
// row (PAGED: the pool page's row).  Runs of tokens inside one page
// are contiguous rows in every layout.
__device__ __forceinline__ void tok_loc(const Geom& g, int b, int t, int* pb, int64_t* row) {
  if (g.layout == KVQ_LAYOUT_PAGED) {
    *pb = 0;
    *row = (int64_t)g.page_table[b * g.max_pages + (t >> kPageShift)] * kPageTok +
           (t & (kPageTok - 1));
  } else {
    *pb = b;
    *row = t;
  }
}
template <typename T>
__device__ __forceinline__ T* tok_ptr(const Geom& g, int which, int b, int h, int t,
                                      int64_t col = 0) {
  int pb;
  int64_t row;
  tok_loc(g, b, t, &pb, &row);
  return plane_ptr<T>(g, which, pb, h, row, col);
}
// Row of 32-token block k of sequence b in a per-block plane (KIVI's key
// scales and zero points; a page holds kPageTok / 32 block rows).
__device__ __forceinline__ void blk_loc(const Geom& g, int b, int k, int* pb, int64_t* row) {
  constexpr int per = kPageTok / 32;
  if (g.layout == KVQ_LAYOUT_PAGED) {
    *pb = 0;
    *row = (int64_t)g.page_table[b * g.max_pages + k / per] * per + k % per;
  } else {
    *pb = b;
    *row = k;
  }
}
template <typename T>
__device__ __forceinline__ T* blk_ptr(const Geom& g, int which, int b, int h, int k,
                                      int64_t col = 0) {
  int pb;
  int64_t row;
  blk_loc(g, b, k, &pb, &row);
  return plane_ptr<T>(g, which, pb, h, row, col);
}

// Device address of the library's error word (set up once per device).
int* device_error_word();

// Bytes of the device state region at the start of a cache buffer (zeroed
// on the first launch after create/reset): the CacheState block, one split
// arrival counter per (sequence, kv head), then for RAGGED / PAGED layouts
// seq_len[B], seq_new[B] and the page table [B][max_pages].
inline size_t state_region_bytes(int B, int H, int layout = KVQ_LAYOUT_UNIFORM,
                                 int max_pages = 0) {
  auto a256 = [](size_t x) { return (x + 255) & ~size_t(255); };
  size_t n = sizeof(CacheState) + a256((size_t)B * H * 4);
  if (layout != KVQ_LAYOUT_UNIFORM) n += a256((size_t)2 * B * 4);
  if (layout == KVQ_LAYOUT_PAGED) n += a256((size_t)B * max_pages * 4);
  return n;
}
inline size_t state_region_bytes(const Geom& g) {
  return state_region_bytes(g.B, g.H, g.layout, g.max_pages);
}

// Floats of split-K partials a decode over this geometry addresses:
// [B][Hq][kMaxSplits][D + kWsStride].
inline size_t workspace_floats(const Geom& g) {
  return (size_t)g.B * g.Hq * kMaxSplits * (g.D + kWsStride);
}

// Record a failure for kvq_last_error() and return `st`.
kvq_status set_error(kvq_status st, const char* fmt, ...);

int num_sms();

}  // namespace kvq

// Host-side handle of a cache (opaque to users of kvq.h).
struct kvq_cache {
  kvq_cache_desc desc;
  kvq::Geom g;
  char* base;
  size_t bytes;
  int T;            // host mirror of the device token count (RAGGED / PAGED: max T_b)
  bool need_init;   // device state not yet zeroed since create/reset
  bool need_clear;  // workspace and epoch not yet zeroed since create
  // RAGGED / PAGED: host mirrors of the per-sequence counts; PAGED: each
  // sequence's pool pages in token order and the pool's free list
  std::vector<int> seq_T, seq_n;
  std::vector<std::vector<int>> seq_pages;
  std::vector<int> free_pages;
};

namespace kvq {
// Zero the cache's device state if this is the first launch since
// create/reset (stream-ordered memset).
cudaError_t ensure_cache_init(kvq_cache* c, cudaStream_t s);
}  // namespace kvq
