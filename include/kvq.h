/*
 * kvq — packed low-bit KV-cache attention step with LoRA-adapted Q/K/V
 * projections, for NVIDIA GB300 (sm_103a).  C ABI.
 *
 * The step follows "Quality Recovery for Quantized KV Caches via Low-Rank
 * Attention Adaptation" (arXiv 2609.04263):
 *   kvq_project_lora    Section 3, Eq. (1) and Eq. (lora): Q/K/V = H W'^T with
 *                       W' = W + (alpha/r) B A, kept as an explicit rank-r
 *                       branch (Section 3.4), then rotary positions on Q, K.
 *   kvq_append_pack     Section 3.1, Eq. (affine) and the symmetric control;
 *                       KIVI and KVarN formats: new keys/values are coded and
 *                       appended; no unquantized copy is kept beyond the
 *                       format's own full-precision window.
 *   kvq_attend_prefill  Sections 3.1-3.3: causal attention of the newly
 *   kvq_attend_decode   appended tokens over the stored reconstruction
 *                       R_phi(K, V) of every cached token.
 *   kvq_attend_backward Section 3.3: straight-through backward (x_hat + x -
 *   kvq_lora_backward   stopgrad(x)) through attention into the adapters.
 *
 * Conventions for every call:
 *   - Tensor arguments are DEVICE pointers owned by the caller, row-major and
 *     contiguous.  The library never allocates device memory: a cache lives
 *     in a caller-provided buffer of kvq_cache_bytes() bytes.
 *   - `stream` is a cudaStream_t (NULL = legacy default stream).  Calls are
 *     asynchronous on that stream; the caller orders calls on one cache.
 *   - Arguments are validated on the host before anything is launched; a
 *     failed validation returns a status, launches nothing and leaves the
 *     cache unchanged.  kvq_last_error() describes the last failure of the
 *     calling thread.
 *   - Inputs must be finite.
 *   - The dtype (KVQ_F32 or KVQ_BF16) is the activation dtype: it applies to
 *     hidden states, weights, LoRA factors, q/k/v, outputs and the
 *     full-precision cache windows.  Accumulation is fp32; cache metadata is
 *     fp16.
 */
#ifndef KVQ_H
#define KVQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define KVQ_ABI_VERSION 1

typedef enum {
  KVQ_OK = 0,
  KVQ_ERR_ARG = 1,          /* null pointer, bad enum, negative size         */
  KVQ_ERR_SHAPE = 2,        /* inconsistent or unsupported dimensions        */
  KVQ_ERR_CAPACITY = 3,     /* append beyond max_tokens, buffer too small    */
  KVQ_ERR_UNSUPPORTED = 4,  /* format/bit-width/dtype combination not built  */
  KVQ_ERR_CUDA = 5,         /* a CUDA launch or query failed                 */
  KVQ_ERR_TIMEOUT = 6       /* a bounded device-side wait gave up            */
} kvq_status;

/* Cache formats (Section 3.1). */
typedef enum {
  KVQ_FMT_FLOAT = 0,      /* control: K/V stored in the activation dtype        */
  KVQ_FMT_AFFINE = 1,     /* Eq. (affine): groups of `group_size` along D, codes
                             round((x - min)/s), fp16 scale and fp16 offset     */
  KVQ_FMT_SYMMETRIC = 2,  /* maximum-magnitude fp16 scale, no offset; signed
                             code q in [-(2^(b-1)-1), 2^(b-1)-1] stored as
                             q + 2^(b-1)                                        */
  KVQ_FMT_KIVI = 3,       /* keys per channel (group = 32-token block x one
                             channel), values per token (groups along D), the
                             newest R..R+G-1 tokens kept at full precision      */
  KVQ_FMT_KVARN = 4       /* first `sink_tokens` kept at full precision; then
                             blocks of `group_size` tokens: normalised Hadamard
                             on D, `norm_iters` rounds of dual-axis variance
                             normalisation, grouped affine codes                */
} kvq_format;

typedef enum { KVQ_F32 = 0, KVQ_BF16 = 1 } kvq_dtype;

/* Geometry and format of one layer's cache. */
typedef struct {
  int32_t fmt;              /* kvq_format                                       */
  int32_t key_bits;         /* 2, 4 or 8 (ignored for FLOAT)                     */
  int32_t value_bits;       /* 2, 4 or 8 (ignored for FLOAT)                     */
  int32_t group_size;       /* G: divides head_dim; KIVI/KVarN: also the token
                               block length (power of two for KVarN)            */
  int32_t residual_tokens;  /* KIVI: R (>= 0)                                    */
  int32_t sink_tokens;      /* KVarN: S (>= 0)                                   */
  int32_t norm_iters;       /* KVarN: normalisation iterations (paper: 8)        */
  int32_t batch;            /* B sequences (layout UNIFORM: all holding the same
                               token count)                                      */
  int32_t kv_heads;         /* Hkv                                               */
  int32_t q_heads;          /* Hq (multiple of Hkv); sizes the decode workspace */
  int32_t head_dim;         /* D: 64, 128 or 256                                 */
  int32_t max_tokens;       /* capacity per sequence                             */
  int32_t dtype;            /* kvq_dtype of the full-precision windows           */
  int32_t layout;           /* kvq_layout (0 = UNIFORM)                          */
  int32_t num_pages;        /* layout PAGED: pages of KVQ_PAGE_TOKENS tokens in
                               the pool shared by all sequences                 */
} kvq_cache_desc;

/* Token layout of a cache.
 *   UNIFORM  every sequence holds the same number of tokens T (appends add L
 *            tokens to all of them).
 *   RAGGED   every sequence b has its own count T_b <= max_tokens, in its own
 *            rows (continuous batching: sequences start, grow and are
 *            released independently).
 *   PAGED    RAGGED, with each sequence's tokens in pages of KVQ_PAGE_TOKENS
 *            tokens taken from one pool of num_pages pages by the library's
 *            allocator as the sequence grows, and returned by
 *            kvq_seq_release; a sequence holds ceil(T_b / 256) pages.
 * RAGGED and PAGED caches are built for bf16 AFFINE, SYMMETRIC and KIVI caches
 * with group_size 32, key_bits == value_bits in {2, 4}, head_dim 64 or 128, at
 * most 16 query heads per kv head and at most KVQ_MAX_SEQS sequences (KIVI's
 * residual ring stays per sequence; its coded blocks go to pages). */
typedef enum { KVQ_LAYOUT_UNIFORM = 0, KVQ_LAYOUT_RAGGED = 1, KVQ_LAYOUT_PAGED = 2 } kvq_layout;
#define KVQ_PAGE_TOKENS 256
#define KVQ_MAX_SEQS 512

typedef struct kvq_cache kvq_cache;   /* opaque, host-side bookkeeping only */

/* Planes of a cache, for inspection and tests (kvq_cache_view). */
enum {
  KVQ_PLANE_K_CODES = 0,  /* uint8 [B][Hkv][rows][D*kb/8], LSB-first bit order   */
  KVQ_PLANE_K_SCALE,      /* fp16: per token [rows][D/G]; KIVI [blocks][D]       */
  KVQ_PLANE_K_ZERO,       /* fp16, same shape as K_SCALE (affine formats)        */
  KVQ_PLANE_V_CODES,
  KVQ_PLANE_V_SCALE,
  KVQ_PLANE_V_ZERO,
  KVQ_PLANE_K_FULL,       /* act dtype: FLOAT all tokens; KIVI residual ring of
                             R+G slots (token t in slot t mod (R+G)); KVarN sinks */
  KVQ_PLANE_V_FULL,
  KVQ_PLANE_K_PEND,       /* act dtype, KVarN staging ring [G][D], slot (t-S) mod G */
  KVQ_PLANE_V_PEND,
  KVQ_PLANE_K_ROW,        /* fp16 KVarN row scales, one per quantized token      */
  KVQ_PLANE_K_COL,        /* fp16 KVarN column scales [blocks][D]                */
  KVQ_PLANE_V_ROW,
  KVQ_PLANE_V_COL,
  KVQ_PLANE_WORKSPACE,    /* fp32 decode split-K partials (not cache state)      */
  KVQ_NUM_PLANES
};

typedef struct {
  void* ptr[KVQ_NUM_PLANES];          /* device pointer, NULL if absent        */
  int64_t dims[KVQ_NUM_PLANES][4];    /* [B][Hkv][rows][cols], row-major       */
  int32_t elem_bytes[KVQ_NUM_PLANES]; /* 1 codes, 2 fp16/bf16, 4 fp32           */
  int32_t tokens;                     /* T: tokens stored per sequence          */
  int32_t quantized_tokens;           /* tokens held as codes (KIVI/KVarN: the
                                         quantized prefix; AFFINE/SYM: T)      */
} kvq_cache_planes;

/* Device bytes a cache with this descriptor needs (0 if the descriptor is
 * invalid; see kvq_last_error). */
size_t kvq_cache_bytes(const kvq_cache_desc* desc);

/* Bind a cache to `dev_buf` (caller-owned, >= kvq_cache_bytes, 256-byte
 * aligned).  Allocates only the host-side handle; the buffer contents need no
 * initialisation (the first launching call zeroes the cache's 256-byte device
 * state block on its stream).  The cache starts empty (T = 0).
 *
 * The token count T lives in device memory and kernels read it there, so a
 * sequence of calls can be captured into a CUDA graph and replayed: every
 * replayed append advances T on the device.  The host keeps a mirror for
 * argument checks; after replays, kvq_cache_sync() refreshes it. */
kvq_status kvq_create_cache(const kvq_cache_desc* desc, void* dev_buf, size_t bytes,
                            kvq_cache** out);

/* Free the host handle.  The device buffer stays the caller's. */
kvq_status kvq_destroy_cache(kvq_cache* cache);

/* Forget every stored token.  Nothing is launched here: the device state is
 * zeroed, on the caller's stream, by the next launching call. */
kvq_status kvq_reset_cache(kvq_cache* cache);

/* Tokens stored per sequence according to the host mirror, -1 for NULL. */
int kvq_cache_tokens(const kvq_cache* cache);

/* Read the device token count into the host mirror (synchronises `stream`).
 * Returns KVQ_ERR_CAPACITY (and clears the flag) if a replayed append was
 * refused on the device because it would exceed max_tokens; a refused
 * append writes nothing and leaves T unchanged. */
kvq_status kvq_cache_sync(kvq_cache* cache, void* stream);

/* Device pointers and shapes of every plane (for tests and export). */
kvq_status kvq_cache_view(const kvq_cache* cache, kvq_cache_planes* out);

/*
 * Q/K/V projection with explicit LoRA branches and rotary positions
 * (Section 3, Eq. 1 and Eq. lora; cost per token per Section 3.4).
 *
 *   x       [B][L][d_in]                     hidden states
 *   w_qkv   [(Hq + 2 Hkv) * D][d_in]          frozen W_Q, W_K, W_V stacked by rows
 *   a_p     [r_p][d_in], b_p [d_out_p][r_p]   LoRA factors of p in {q,k,v};
 *                                             r_p = 0 (pointers ignored) means no
 *                                             adapter on p (placements Q/K/QK/QKV)
 *   out     q [B][Hq][L][D], k and v [B][Hkv][L][D]   (head-major)
 *
 *   y_p = x W_p^T + alpha_over_r * (x A_p^T) B_p^T, then rotate-half RoPE on
 *   q and k at positions P + pos0 + l with frequencies rope_base^(-2i/D)
 *   (rope_base = 0 disables RoPE), where P = 0 if pos_cache is NULL, else the
 *   token count of pos_cache read on the device when the kernel runs (the
 *   usual choice: new tokens continue the cached sequence, and a captured
 *   decode step stays correct on replay).  r_p <= 64, multiple of 8 for
 *   KVQ_BF16.  d_in must be a multiple of 64 for KVQ_BF16.
 */
kvq_status kvq_project_lora(const void* x, int B, int L, int d_in, const void* w_qkv,
                            const void* a_q, const void* b_q, int r_q,
                            const void* a_k, const void* b_k, int r_k,
                            const void* a_v, const void* b_v, int r_v,
                            float alpha_over_r, int n_q_heads, int n_kv_heads,
                            int head_dim, int pos0, kvq_cache* pos_cache, float rope_base,
                            int dtype, void* q, void* k, void* v, void* stream);

/*
 * kvq_project_lora over a frozen NF4 base (Sections 3.4 and 4: the reported
 * Gemma and Llama-3.1 runs keep NF4 bases with explicit rank-r branches;
 * Section 2 cites QLoRA's 4-bit NormalFloat data type for them).  bf16 only.
 *
 *   w_codes   uint8 [(Hq + 2 Hkv) * D][d_in / 2]: 4-bit NF4 codes, input k of a
 *             row in byte k / 2 (even k in the low nibble)
 *   w_absmax  float [(Hq + 2 Hkv) * D][d_in / 64]: one scale per block of 64
 *             consecutive inputs (4-byte aligned)
 *   a base weight is level[code] * absmax, with the 16 NF4 levels of QLoRA;
 *   every other argument as in kvq_project_lora.
 *
 * The base is dequantized inside the GEMM (per 64-input tile, into shared
 * memory as bf16) and never materialised in device memory.  KVQ_ERR_UNSUPPORTED
 * unless d_in % 64 == 0, head_dim is 64 or 128, Hq * D and Hkv * D are
 * multiples of 128, and the ranks are multiples of 8 up to 64.
 */
kvq_status kvq_project_lora_nf4(const void* x, int B, int L, int d_in, const void* w_codes,
                                const void* w_absmax, const void* a_q, const void* b_q, int r_q,
                                const void* a_k, const void* b_k, int r_k,
                                const void* a_v, const void* b_v, int r_v,
                                float alpha_over_r, int n_q_heads, int n_kv_heads, int head_dim,
                                int pos0, kvq_cache* pos_cache, float rope_base, void* q, void* k,
                                void* v, void* stream);

/*
 * Projection of L new tokens per sequence fused with their append (Section 3,
 * Eq. (1) and Eq. (lora), then Section 3.1: the new keys and values are coded
 * into the packed cache straight from the projection, without an unquantized
 * copy in device memory).
 *
 *   x      [B][L][d_in] hidden states, B the cache's batch
 *   w_qkv, a_p, b_p, r_p, alpha_over_r, rope_base  as in kvq_project_lora; the
 *          projection dimensions are the cache's (Hq, Hkv, head_dim)
 *   q      [B][Hq][L][D] receives the rotated queries
 *
 * Keys (after RoPE) and values are rounded to bf16, exactly the values
 * kvq_project_lora would store, and coded per token into the cache at
 * positions T .. T + L - 1 (T = the cache's device token count, which the call
 * then advances by L): the cache after the call is bit for bit the cache
 * kvq_project_lora + kvq_append_pack would leave.  Covered shapes
 * (kvq_project_append_supported tells): bf16 affine or symmetric caches with
 * group size 32 and 2/4/8-bit codes, B * L > 16 rows, d_in a multiple of 64,
 * head counts that tile the tensor-core projection, ranks multiples of 8 up to
 * 64.  Otherwise KVQ_ERR_UNSUPPORTED and nothing is launched: use the two calls.
 * KVQ_ERR_CAPACITY if T + L > max_tokens (host mirror; a replayed call that
 * would overflow is refused on the device like an append).
 */
kvq_status kvq_project_append(kvq_cache* cache, const void* x, int L, int d_in,
                              const void* w_qkv, const void* a_q, const void* b_q, int r_q,
                              const void* a_k, const void* b_k, int r_k,
                              const void* a_v, const void* b_v, int r_v,
                              float alpha_over_r, float rope_base, void* q, void* stream);

/* 1 when kvq_project_append covers this cache, L, d_in and ranks, 0 when it
 * does not, -1 for a NULL cache.  Launches nothing. */
int kvq_project_append_supported(const kvq_cache* cache, int L, int d_in, int r_q, int r_k,
                                 int r_v);

/*
 * Append L new tokens per sequence: k, v [B][Hkv][L][D] (activation dtype).
 * Codes them per the cache format (Section 3.1) into the packed planes.  The
 * cache after T tokens is the same whether they arrive in one call or in
 * chunks.  KVQ_ERR_CAPACITY if T + L > max_tokens (host mirror); the kernels
 * check the device count again and refuse an overflowing replayed append.
 * KVQ_ERR_SHAPE if B * Hkv exceeds 65535, or if B * Hkv * (L + group_size) *
 * D / 4 reaches 2^31 (the kernels index one call's elements in 32 bits):
 * append such a span in chunks instead.
 */
kvq_status kvq_append_pack(kvq_cache* cache, const void* k, const void* v, int L,
                           void* stream);

/*
 * Causal attention of the L most recently appended tokens' queries over the
 * reconstruction of all T cached tokens (Sections 3.2-3.3).  Query l sits at
 * position T - L + l and sees tokens 0 .. T - L + l.  q, out [B][Hq][L][D];
 * query head h reads kv head h / (Hq / Hkv).  softmax_scale is usually
 * 1/sqrt(D).  Must follow kvq_append_pack of the same L tokens.
 */
kvq_status kvq_attend_prefill(kvq_cache* cache, const void* q, int L, int n_q_heads,
                              float softmax_scale, void* out, void* stream);

/*
 * Decode step: kvq_attend_prefill with L = 1, split over the tokens across
 * thread blocks with a log-sum-exp merge (partials in the cache's workspace
 * plane, so calls on one cache must not overlap).  q, out [B][Hq][1][D].
 */
kvq_status kvq_attend_decode(kvq_cache* cache, const void* q, int n_q_heads,
                             float softmax_scale, void* out, void* stream);

/*
 * One decode step of one layer: kvq_project_lora of the new token (x [B][1]
 * [d_in], positions continue the cache), kvq_append_pack of its key and value,
 * then kvq_attend_decode of its query (Sections 3-3.3).  q, k, v receive the
 * projections ([B][Hq][1][D], [B][Hkv][1][D] x 2); out [B][Hq][1][D].  B and
 * the head counts are the cache's.  For bf16 affine/symmetric caches with
 * 2/4-bit codes, G = 32, head_dim 64/128, B <= 16, d_in a multiple of 256 and
 * ranks that are multiples of 8 up to 64 (kvq_decode_step_fused tells) the
 * three steps run as one cooperative kernel with one CTA per SM, whose CTAs
 * hand results to one another through the cache's workspace with bounded
 * waits; other shapes run the three calls in order.  Both give the same codes
 * for the same k and v and agree to bf16 rounding.  Like kvq_attend_decode
 * it uses the cache's workspace, so calls on one cache must not overlap.
 * The fused kernel starts reading w_qkv and the LoRA factors before the work
 * queued before it on `stream` has finished (programmatic dependent launch):
 * that work must not write them.
 */
kvq_status kvq_decode_step(kvq_cache* cache, const void* x, int d_in, const void* w_qkv,
                           const void* a_q, const void* b_q, int r_q,
                           const void* a_k, const void* b_k, int r_k,
                           const void* a_v, const void* b_v, int r_v,
                           float alpha_over_r, float rope_base, float softmax_scale,
                           void* q, void* k, void* v, void* out, void* stream);

/*
 * 1 when kvq_decode_step on `cache` with this d_in and these LoRA ranks runs
 * as the one fused kernel, 0 when it runs the three separate calls, -1 when
 * cache is NULL.  Launches nothing.
 */
int kvq_decode_step_fused(const kvq_cache* cache, int d_in, int r_q, int r_k, int r_v);

/*
 * kvq_attend_decode for callers that cannot allocate device memory.  (No
 * counterpart in the paper: this is a deployment variant of the decode step.)
 *
 * kvq_attend_decode keeps its split-K partials in the cache buffer's
 * workspace plane.  Callers that cannot provide extra device memory when they
 * call (a plugin or custom-op host that passes only input and output tensors
 * and forbids allocation, allocation-free serving loops where cudaMalloc
 * would synchronise the device, a process whose memory pool has reserved all
 * free HBM) use this variant instead: the partials go to one fixed array in
 * the library's static device memory (4 MiB per GPU, held from library load
 * until process exit), and the call allocates nothing.
 *
 * Same arguments, semantics and results as kvq_attend_decode.  Returns
 * KVQ_ERR_CAPACITY, launching nothing, if batch * q_heads * 32 * (head_dim + 2)
 * floats exceed the array (1,048,576 floats).  The first call on each device
 * looks up the array's device address with that device current; make that
 * first call before any stream capture.  The address is kept for the life of
 * the process: do not use the library on a device after cudaDeviceReset().
 * Every call uses the same array and
 * leaves its contents behind (the kernels write every partial they later
 * read, so nothing needs clearing), so calls that overlap on the GPU (other
 * streams, other threads) race: serialise them.
 */
kvq_status kvq_attend_decode_noalloc(kvq_cache* cache, const void* q, int n_q_heads,
                                     float softmax_scale, void* out, void* stream);

/*
 * Backward of attention over the stored reconstruction (Section 3.3): the
 * gradients of sum(out * d_out) for out = kvq_attend_prefill(q) of the L
 * newest queries over all T cached tokens.  Appended states enter attention
 * as x_hat + x - stopgrad(x) (the straight-through estimator), so d_k and d_v,
 * the gradients at the reconstruction x_hat, are also the gradients of the
 * keys and values that were coded into the cache, and feed the K and V
 * adapters unchanged (kvq_lora_backward).
 *   q, d_out  [B][Hq][L][D] in the cache's dtype (d_out: gradient of out)
 *   d_q       [B][Hq][L][D] fp32
 *   d_k, d_v  [B][Hkv][T][D] fp32 (every query head of a kv head's group
 *             summed; tokens no query sees get 0)
 * workspace: caller-owned device memory, at least
 * kvq_attend_backward_workspace() bytes (one (sequence, kv head) pair's fp32
 * reconstruction, scores and score gradients); a larger workspace processes
 * that many pairs per pass.  Formats FLOAT, AFFINE, SYMMETRIC and KIVI;
 * KVarN returns KVQ_ERR_UNSUPPORTED.  Too small a workspace returns
 * KVQ_ERR_CAPACITY.  The cache is not modified.
 */
size_t kvq_attend_backward_workspace(const kvq_cache* cache, int L, int n_q_heads);
kvq_status kvq_attend_backward(kvq_cache* cache, const void* q, const void* d_out, int L,
                               int n_q_heads, float softmax_scale, float* d_q, float* d_k,
                               float* d_v, void* workspace, size_t workspace_bytes,
                               void* stream);

/*
 * Backward of kvq_project_lora into its rank-r factors (Eq. (1), Eq. (lora),
 * Section 3.4: the base W stays frozen).  d_q [B][Hq][L][D], d_k and d_v
 * [B][Hkv][kv_rows][D] (fp32) are gradients of the projection's outputs after
 * RoPE; the last L of each head's kv_rows rows belong to the L tokens of x
 * (kv_rows = T passes kvq_attend_backward's d_k, d_v directly when the cache
 * holds x's tokens last).  Writes, in fp32:
 *   da_p [r_p][d_in] = (alpha/r) (g_p B_p)^T x,  db_p [n_p][r_p] = (alpha/r) g_p^T (x A_p^T)
 * where g_p is the gradient before RoPE, and, if d_x is not NULL,
 *   d_x [B][L][d_in] = g W + sum_p (alpha/r) (g_p B_p) A_p   (needs w_qkv).
 * x, w_qkv and the factors are in `dtype`, laid out as for kvq_project_lora;
 * a projection with r_p = 0 has no factors and its gradients are not written.
 * With bf16 activations, d_in a multiple of 128 and (Hq + 2 Hkv) D a multiple of
 * 64, g W runs on the tensor cores: g is split in the workspace into bf16 high and
 * low parts (about 16 significant bits) against W^T, which the call also writes
 * into the workspace.
 * workspace: at least kvq_lora_backward_workspace() bytes (a function of the
 * shape alone; 16-byte aligned).
 */
size_t kvq_lora_backward_workspace(int B, int L, int d_in, int n_q_heads, int n_kv_heads,
                                   int head_dim, int r_q, int r_k, int r_v);
kvq_status kvq_lora_backward(const void* x, int B, int L, int d_in, const void* w_qkv,
                             const void* a_q, const void* b_q, int r_q,
                             const void* a_k, const void* b_k, int r_k,
                             const void* a_v, const void* b_v, int r_v,
                             float alpha_over_r, int n_q_heads, int n_kv_heads, int head_dim,
                             int pos0, float rope_base, int dtype,
                             const float* d_q, const float* d_k, const float* d_v, int kv_rows,
                             float* da_q, float* db_q, float* da_k, float* db_k,
                             float* da_v, float* db_v, float* d_x,
                             void* workspace, size_t workspace_bytes, void* stream);

/*
 * Ragged appends (layouts RAGGED and PAGED): sequence b appends the first
 * n[b] (0 <= n[b] <= L) of its L rows of k, v [B][Hkv][L][D] at its own
 * positions T_b .. T_b + n[b] - 1.  n is a HOST array of B counts; NULL means
 * n[b] = L for every b (kvq_append_pack on a ragged cache does the same).
 * A PAGED cache first takes the pages the new tokens need from its pool;
 * KVQ_ERR_CAPACITY (nothing appended, no page taken) if some T_b + n[b]
 * exceeds max_tokens or the pool runs out.  kvq_attend_prefill and
 * kvq_attend_decode then attend, per sequence, the n[b] rows of the last
 * append (prefill: rows l < n[b] of q and out; the rest of out is not
 * written) or its newest token (decode; a sequence holding no token gets a
 * zero output) over that sequence's T_b tokens.  A PAGED append that takes
 * new pages copies their table entries from host memory on `stream`, so it
 * must not be captured in a CUDA graph; RAGGED appends and the attention
 * calls can be (kvq_cache_sync then refreshes the host's per-sequence counts).
 */
kvq_status kvq_append_pack_ragged(kvq_cache* cache, const void* k, const void* v, int L,
                                  const int* n, void* stream);

/* Tokens held by sequence b (any layout; -1 for a bad argument). */
int kvq_seq_tokens(const kvq_cache* cache, int b);

/* Layouts RAGGED and PAGED: sequence b becomes empty (T_b = 0) and a PAGED
 * cache returns its pages to the pool.  Stream-ordered like an append. */
kvq_status kvq_seq_release(kvq_cache* cache, int b, void* stream);

/* Pages of a PAGED cache's pool not held by any sequence (-1 otherwise). */
int kvq_free_pages(const kvq_cache* cache);

/* PAGED: the pool pages of sequence b in token order (page i holds its tokens
 * 64 i .. 64 i + 63; in kvq_cache_view's planes a page is rows 64 p .. 64 p +
 * 63 of batch index 0).  Writes at most max_pages ids to pages and returns
 * the sequence's page count, or -1. */
int kvq_seq_pages(const kvq_cache* cache, int b, int* pages, int max_pages);

/* Read and clear the device-side error word of the library (synchronises
 * `stream`).  *out = 0 when no bounded wait has timed out; otherwise a kernel
 * gave up waiting (a TMA ring, a handoff between CTAs, a merge), returned
 * early and left its output incomplete, and KVQ_ERR_TIMEOUT is returned.  The
 * word's address is looked up once per device: do not use the library on a
 * device after cudaDeviceReset(). */
kvq_status kvq_device_status(void* stream, int* out);

/* Description of the last failure on this thread ("" if none). */
const char* kvq_last_error(void);

/* KVQ_ABI_VERSION of the loaded library. */
int kvq_abi_version(void);

#ifdef __cplusplus
}
#endif
#endif /* KVQ_H */
