// C-ABI entry points: argument validation, cache geometry and bookkeeping.
// Kernels live in pack.cu, attend.cu and project.cu.
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <algorithm>
#include <mutex>
#include <string>
#include <vector>

#include "kvq_internal.cuh"

using namespace kvq;

namespace {

thread_local std::string g_last_error;

kvq_status vfail(kvq_status st, const char* fmt, va_list ap) {
  char buf[512];
  vsnprintf(buf, sizeof buf, fmt, ap);
  g_last_error = buf;
  return st;
}

kvq_status fail(kvq_status st, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vfail(st, fmt, ap);
  va_end(ap);
  return st;
}

kvq_status cuda_fail(cudaError_t e, const char* where) {
  return fail(KVQ_ERR_CUDA, "%s: %s", where, cudaGetErrorString(e));
}

bool misaligned(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) != 0; }

bool valid_bits(int b) { return b == 2 || b == 4 || b == 8; }
bool pow2(int x) { return x > 0 && (x & (x - 1)) == 0; }

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

// Validate a descriptor and lay out its planes.  Offsets are relative to the
// buffer start; returns the total size, or 0 with g_last_error set.
size_t layout(const kvq_cache_desc* d, Geom* g, size_t off[KVQ_NUM_PLANES],
              kvq_status* st) {
  *st = KVQ_ERR_ARG;
  if (!d) { fail(KVQ_ERR_ARG, "descriptor is NULL"); return 0; }
  if (d->fmt < KVQ_FMT_FLOAT || d->fmt > KVQ_FMT_KVARN) {
    fail(KVQ_ERR_ARG, "unknown format %d", d->fmt); return 0;
  }
  if (d->dtype != KVQ_F32 && d->dtype != KVQ_BF16) {
    fail(KVQ_ERR_ARG, "unknown dtype %d", d->dtype); return 0;
  }
  *st = KVQ_ERR_SHAPE;
  if (d->batch <= 0 || d->kv_heads <= 0 || d->q_heads <= 0 || d->max_tokens <= 0) {
    fail(KVQ_ERR_SHAPE, "batch, kv_heads, q_heads and max_tokens must be positive"); return 0;
  }
  if (d->q_heads % d->kv_heads != 0) {
    fail(KVQ_ERR_SHAPE, "q_heads %d is not a multiple of kv_heads %d", d->q_heads, d->kv_heads);
    return 0;
  }
  if (d->q_heads / d->kv_heads > 16) {
    fail(KVQ_ERR_UNSUPPORTED, "GQA group %d > 16", d->q_heads / d->kv_heads);
    *st = KVQ_ERR_UNSUPPORTED; return 0;
  }
  if (d->head_dim != 64 && d->head_dim != 128 && d->head_dim != 256) {
    fail(KVQ_ERR_UNSUPPORTED, "head_dim %d (supported: 64, 128, 256)", d->head_dim);
    *st = KVQ_ERR_UNSUPPORTED; return 0;
  }
  const int D = d->head_dim, G = d->group_size;
  if (d->fmt != KVQ_FMT_FLOAT) {
    if (!valid_bits(d->key_bits) || !valid_bits(d->value_bits)) {
      fail(KVQ_ERR_UNSUPPORTED, "bit widths %d/%d (supported: 2, 4, 8)", d->key_bits,
           d->value_bits);
      *st = KVQ_ERR_UNSUPPORTED; return 0;
    }
    if (G < 8 || !pow2(G) || D % G != 0 || G > D) {
      fail(KVQ_ERR_SHAPE, "group_size %d must be a power of two in [8, head_dim] dividing %d",
           G, D);
      return 0;
    }
  }
  if (d->fmt == KVQ_FMT_KIVI && d->residual_tokens < 0) {
    fail(KVQ_ERR_SHAPE, "residual_tokens must be >= 0"); return 0;
  }
  if (d->fmt == KVQ_FMT_KVARN) {
    if (d->sink_tokens < 0 || d->norm_iters < 0 || d->norm_iters > 64) {
      fail(KVQ_ERR_SHAPE, "sink_tokens >= 0 and 0 <= norm_iters <= 64 required"); return 0;
    }
    if (G > 128 || G * D > 16384) {
      fail(KVQ_ERR_UNSUPPORTED, "KVarN block of %d tokens x %d channels (max 128 tokens, "
           "16384 elements)", G, D);
      *st = KVQ_ERR_UNSUPPORTED; return 0;
    }
  }
  if (d->layout < KVQ_LAYOUT_UNIFORM || d->layout > KVQ_LAYOUT_PAGED) {
    fail(KVQ_ERR_ARG, "unknown layout %d", d->layout); *st = KVQ_ERR_ARG; return 0;
  }
  if (d->layout != KVQ_LAYOUT_UNIFORM) {
    const bool ok = (d->fmt == KVQ_FMT_AFFINE || d->fmt == KVQ_FMT_SYMMETRIC ||
                     d->fmt == KVQ_FMT_KIVI) &&
                    d->dtype == KVQ_BF16 && G == 32 && d->key_bits == d->value_bits &&
                    (d->key_bits == 2 || d->key_bits == 4) && (D == 64 || D == 128) &&
                    d->q_heads / d->kv_heads <= 16;
    if (!ok) {
      fail(KVQ_ERR_UNSUPPORTED, "ragged and paged layouts need a bf16 affine, symmetric or KIVI "
           "cache with group_size 32, key_bits == value_bits in {2, 4} and head_dim 64 or 128");
      *st = KVQ_ERR_UNSUPPORTED; return 0;
    }
    if (d->batch > KVQ_MAX_SEQS) {
      fail(KVQ_ERR_UNSUPPORTED, "%d sequences > %d", d->batch, KVQ_MAX_SEQS);
      *st = KVQ_ERR_UNSUPPORTED; return 0;
    }
    if (d->layout == KVQ_LAYOUT_PAGED && d->num_pages <= 0) {
      fail(KVQ_ERR_SHAPE, "a paged cache needs num_pages > 0"); return 0;
    }
  }
  const int B = d->batch, H = d->kv_heads, Tm = d->max_tokens;
  const bool paged = d->layout == KVQ_LAYOUT_PAGED;
  // per-token planes hold whole 64-token chunks (the decode kernel copies
  // whole chunks), so their rows are padded to a multiple of 64; a paged
  // cache's planes hold the page pool of all sequences (batch index 0)
  const int Tp = paged ? d->num_pages * kPageTok : (Tm + 63) / 64 * 64;
  const int act = d->dtype == KVQ_BF16 ? 2 : 4;
  memset(g, 0, sizeof *g);
  g->fmt = d->fmt; g->kb = d->key_bits; g->vb = d->value_bits; g->G = G;
  g->R = d->residual_tokens; g->S = d->sink_tokens; g->iters = d->norm_iters;
  g->B = B; g->H = H; g->Hq = d->q_heads; g->D = D; g->Tmax = Tm; g->act = d->dtype;
  g->ring = d->residual_tokens + G;
  g->layout = d->layout;
  g->max_pages = paged ? (Tm + kPageTok - 1) / kPageTok : 0;
  auto set = [&](int which, int64_t rows, int64_t cols, int elem) {
    g->pl[which].rows = rows; g->pl[which].cols = cols; g->pl[which].elem = elem;
  };
  switch (d->fmt) {
    case KVQ_FMT_FLOAT:
      set(KVQ_PLANE_K_FULL, Tm, D, act);
      set(KVQ_PLANE_V_FULL, Tm, D, act);
      break;
    case KVQ_FMT_AFFINE:
    case KVQ_FMT_SYMMETRIC:
      set(KVQ_PLANE_K_CODES, Tp, D * d->key_bits / 8, 1);
      set(KVQ_PLANE_K_SCALE, Tp, D / G, 2);
      set(KVQ_PLANE_V_CODES, Tp, D * d->value_bits / 8, 1);
      set(KVQ_PLANE_V_SCALE, Tp, D / G, 2);
      if (d->fmt == KVQ_FMT_AFFINE) {
        set(KVQ_PLANE_K_ZERO, Tp, D / G, 2);
        set(KVQ_PLANE_V_ZERO, Tp, D / G, 2);
      }
      break;
    case KVQ_FMT_KIVI: {
      const int64_t nblk = (Tp + G - 1) / G;
      set(KVQ_PLANE_K_CODES, nblk * G, D * d->key_bits / 8, 1);
      set(KVQ_PLANE_K_SCALE, nblk, D, 2);
      set(KVQ_PLANE_K_ZERO, nblk, D, 2);
      set(KVQ_PLANE_V_CODES, nblk * G, D * d->value_bits / 8, 1);
      set(KVQ_PLANE_V_SCALE, nblk * G, D / G, 2);
      set(KVQ_PLANE_V_ZERO, nblk * G, D / G, 2);
      set(KVQ_PLANE_K_FULL, g->ring, D, act);
      set(KVQ_PLANE_V_FULL, g->ring, D, act);
      break;
    }
    case KVQ_FMT_KVARN: {
      const int64_t nblk = Tm > d->sink_tokens ? (Tm - d->sink_tokens) / G : 0;
      const int64_t Q = nblk * G;
      if (d->sink_tokens > 0) {
        set(KVQ_PLANE_K_FULL, d->sink_tokens, D, act);
        set(KVQ_PLANE_V_FULL, d->sink_tokens, D, act);
      }
      set(KVQ_PLANE_K_PEND, G, D, act);
      set(KVQ_PLANE_V_PEND, G, D, act);
      if (nblk > 0) {
        set(KVQ_PLANE_K_CODES, Q, D * d->key_bits / 8, 1);
        set(KVQ_PLANE_K_SCALE, Q, D / G, 2);
        set(KVQ_PLANE_K_ZERO, Q, D / G, 2);
        set(KVQ_PLANE_K_ROW, 1, Q, 2);
        set(KVQ_PLANE_K_COL, nblk, D, 2);
        set(KVQ_PLANE_V_CODES, Q, D * d->value_bits / 8, 1);
        set(KVQ_PLANE_V_SCALE, Q, D / G, 2);
        set(KVQ_PLANE_V_ZERO, Q, D / G, 2);
        set(KVQ_PLANE_V_ROW, 1, Q, 2);
        set(KVQ_PLANE_V_COL, nblk, D, 2);
      }
      break;
    }
  }
  g->splits = decode_splits(*g);
  size_t total = state_region_bytes(*g);     // device state, split counters, ragged arrays
  static_assert(sizeof(CacheState) == 256, "state block is 256 bytes");
  for (int i = 0; i < KVQ_NUM_PLANES; ++i) {
    off[i] = 0;
    if (i == KVQ_PLANE_WORKSPACE) continue;
    Plane& p = g->pl[i];
    if (p.rows == 0) continue;
    off[i] = total;
    total = align256(total + (size_t)plane_batch(*g, i) * H * p.rows * p.cols * p.elem);
  }
  // decode workspace: [B][Hq][kMaxSplits][D + 2] fp32, indexed by q head
  off[KVQ_PLANE_WORKSPACE] = total;
  g->pl[KVQ_PLANE_WORKSPACE].rows = kMaxSplits;
  g->pl[KVQ_PLANE_WORKSPACE].cols = D + kWsStride;
  g->pl[KVQ_PLANE_WORKSPACE].elem = 4;
  total = align256(total + (size_t)B * d->q_heads * kMaxSplits * (D + kWsStride) * 4);
  // epoch block of the fused decode step (256 bytes, never reset)
  total += 256;
  *st = KVQ_OK;
  return total;
}

int g_num_sms = 0;
std::mutex g_mu;

}  // namespace

// ---------------------------------------------------------------------------
// device error word: one int in static device memory, address looked up per
// device on first use
// ---------------------------------------------------------------------------
static __device__ int g_kvq_device_error;

namespace kvq {
int* device_error_word() {
  static int* addr[64] = {nullptr};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  std::lock_guard<std::mutex> lk(g_mu);
  if (!addr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_kvq_device_error) != cudaSuccess) return nullptr;
    addr[dev] = static_cast<int*>(p);
  }
  return addr[dev];
}

// Zero the device state before the first launch after create/reset
// (stream-ordered, so it can be captured with the calls that follow).
cudaError_t ensure_cache_init(kvq_cache* c, cudaStream_t s) {
  if (!c->need_init) return cudaSuccess;
  cudaError_t e = cudaSuccess;
  if (c->need_clear) {
    // once per buffer: the workspace (whose tagged words the fused decode
    // step matches against its epoch) and the epoch block after it
    char* ws = static_cast<char*>(c->g.pl[KVQ_PLANE_WORKSPACE].p);
    e = cudaMemsetAsync(ws, 0, reinterpret_cast<char*>(c->g.epoch) + 256 - ws, s);
    if (e == cudaSuccess) c->need_clear = false;
  }
  if (e == cudaSuccess) e = cudaMemsetAsync(c->g.state, 0, state_region_bytes(c->g), s);
  if (e == cudaSuccess) c->need_init = false;
  return e;
}

kvq_status set_error(kvq_status st, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vfail(st, fmt, ap);
  va_end(ap);
  return st;
}

int num_sms() {
  if (g_num_sms == 0) {
    int dev = 0, n = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    g_num_sms = n > 0 ? n : 148;
  }
  return g_num_sms;
}
}  // namespace kvq

extern "C" {

int kvq_abi_version(void) { return KVQ_ABI_VERSION; }

const char* kvq_last_error(void) { return g_last_error.c_str(); }

size_t kvq_cache_bytes(const kvq_cache_desc* desc) {
  Geom g;
  size_t off[KVQ_NUM_PLANES];
  kvq_status st;
  return layout(desc, &g, off, &st);
}

kvq_status kvq_create_cache(const kvq_cache_desc* desc, void* dev_buf, size_t bytes,
                            kvq_cache** out) {
  if (!out) return fail(KVQ_ERR_ARG, "out is NULL");
  *out = nullptr;
  if (!dev_buf) return fail(KVQ_ERR_ARG, "dev_buf is NULL");
  if (reinterpret_cast<uintptr_t>(dev_buf) % 256 != 0)
    return fail(KVQ_ERR_ARG, "dev_buf must be 256-byte aligned");
  Geom g;
  size_t off[KVQ_NUM_PLANES];
  kvq_status st;
  size_t need = layout(desc, &g, off, &st);
  if (need == 0) return st;
  if (bytes < need)
    return fail(KVQ_ERR_CAPACITY, "buffer of %zu bytes < %zu needed", bytes, need);
  kvq_cache* c = new kvq_cache;
  c->desc = *desc;
  c->g = g;
  c->base = static_cast<char*>(dev_buf);
  c->bytes = bytes;
  c->T = 0;
  c->need_init = true;
  c->need_clear = true;
  c->g.state = reinterpret_cast<CacheState*>(c->base);
  c->g.counters = reinterpret_cast<uint32_t*>(c->base + sizeof(CacheState));
  c->g.epoch = reinterpret_cast<uint32_t*>(c->base + need - 256);
  for (int i = 0; i < KVQ_NUM_PLANES; ++i)
    c->g.pl[i].p = c->g.pl[i].rows ? c->base + off[i] : nullptr;
  c->g.seq_len = c->g.seq_new = c->g.page_table = nullptr;
  if (g.layout != KVQ_LAYOUT_UNIFORM) {
    char* p = c->base + state_region_bytes(g.B, g.H);
    c->g.seq_len = reinterpret_cast<int32_t*>(p);
    c->g.seq_new = c->g.seq_len + g.B;
    if (g.layout == KVQ_LAYOUT_PAGED)
      c->g.page_table = reinterpret_cast<int32_t*>(p + align256((size_t)2 * g.B * 4));
    c->seq_T.assign(g.B, 0);
    c->seq_n.assign(g.B, 0);
    c->seq_pages.assign(g.B, std::vector<int>());
    if (g.layout == KVQ_LAYOUT_PAGED)
      for (int i = desc->num_pages - 1; i >= 0; --i) c->free_pages.push_back(i);
  }
  *out = c;
  g_last_error.clear();
  return KVQ_OK;
}

kvq_status kvq_destroy_cache(kvq_cache* cache) {
  if (!cache) return fail(KVQ_ERR_ARG, "cache is NULL");
  delete cache;
  return KVQ_OK;
}

kvq_status kvq_reset_cache(kvq_cache* cache) {
  if (!cache) return fail(KVQ_ERR_ARG, "cache is NULL");
  cache->T = 0;
  cache->need_init = true;
  if (cache->g.layout != KVQ_LAYOUT_UNIFORM) {
    for (int b = 0; b < cache->g.B; ++b) {
      cache->seq_T[b] = cache->seq_n[b] = 0;
      for (int p : cache->seq_pages[b]) cache->free_pages.push_back(p);
      cache->seq_pages[b].clear();
    }
  }
  return KVQ_OK;
}

static cudaError_t ensure_init(kvq_cache* c, cudaStream_t s) { return ensure_cache_init(c, s); }

kvq_status kvq_cache_sync(kvq_cache* cache, void* stream) {
  if (!cache) return fail(KVQ_ERR_ARG, "cache is NULL");
  cudaStream_t s = (cudaStream_t)stream;
  cudaError_t e = ensure_init(cache, s);
  CacheState st;
  if (e == cudaSuccess) e = cudaMemcpyAsync(&st, cache->g.state, 3 * sizeof(int32_t),
                                            cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e == cudaSuccess && st.error)
    e = cudaMemsetAsync(&cache->g.state->error, 0, sizeof(int32_t), s);
  if (e == cudaSuccess && cache->g.layout != KVQ_LAYOUT_UNIFORM) {
    // per-sequence counts (replayed ragged appends advance them on the device)
    e = cudaMemcpyAsync(cache->seq_T.data(), cache->g.seq_len, cache->g.B * sizeof(int32_t),
                        cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess)
      e = cudaMemcpyAsync(cache->seq_n.data(), cache->g.seq_new, cache->g.B * sizeof(int32_t),
                          cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    int tmax = 0;
    for (int x : cache->seq_T) tmax = std::max(tmax, x);
    st.tokens = tmax;
  }
  if (e != cudaSuccess) return cuda_fail(e, "kvq_cache_sync");
  cache->T = st.tokens;
  if (st.error & kErrCapacity)
    return fail(KVQ_ERR_CAPACITY, "a device-side append was refused: capacity exceeded");
  return KVQ_OK;
}

int kvq_cache_tokens(const kvq_cache* cache) { return cache ? cache->T : -1; }

kvq_status kvq_cache_view(const kvq_cache* cache, kvq_cache_planes* out) {
  if (!cache || !out) return fail(KVQ_ERR_ARG, "cache or out is NULL");
  const Geom& g = cache->g;
  for (int i = 0; i < KVQ_NUM_PLANES; ++i) {
    out->ptr[i] = g.pl[i].p;
    out->dims[i][0] = g.pl[i].rows ? plane_batch(g, i) : 0;
    out->dims[i][1] = g.pl[i].rows ? (i == KVQ_PLANE_WORKSPACE ? g.Hq : g.H) : 0;
    out->dims[i][2] = g.pl[i].rows;
    out->dims[i][3] = g.pl[i].cols;
    out->elem_bytes[i] = g.pl[i].elem;
  }
  out->tokens = cache->T;
  switch (g.fmt) {
    case KVQ_FMT_FLOAT: out->quantized_tokens = 0; break;
    case KVQ_FMT_KIVI: out->quantized_tokens = kivi_tq(cache->T, g.R, g.G); break;
    case KVQ_FMT_KVARN: out->quantized_tokens = kvarn_nblocks(cache->T, g.S, g.G) * g.G; break;
    default: out->quantized_tokens = cache->T;
  }
  return KVQ_OK;
}

kvq_status kvq_append_pack(kvq_cache* cache, const void* k, const void* v, int L,
                           void* stream) {
  if (!cache) return fail(KVQ_ERR_ARG, "cache is NULL");
  if (cache->g.layout != KVQ_LAYOUT_UNIFORM)
    return kvq_append_pack_ragged(cache, k, v, L, nullptr, stream);
  if (L < 0) return fail(KVQ_ERR_ARG, "L = %d < 0", L);
  if (L == 0) return KVQ_OK;
  if (!k || !v) return fail(KVQ_ERR_ARG, "k or v is NULL");
  if (misaligned(k) || misaligned(v)) return fail(KVQ_ERR_ARG, "k and v must be 16-byte aligned");
  if ((int64_t)cache->T + L > cache->g.Tmax)
    return fail(KVQ_ERR_CAPACITY, "append of %d tokens to %d exceeds max_tokens %d", L,
                cache->T, cache->g.Tmax);
  if ((int64_t)cache->g.B * cache->g.H > 65535)
    return fail(KVQ_ERR_SHAPE, "batch x kv heads = %d above 65535",
                cache->g.B * cache->g.H);
  if ((int64_t)cache->g.B * cache->g.H * ((int64_t)L + cache->g.G) * (cache->g.D / 4) >=
      ((int64_t)1 << 31))
    return fail(KVQ_ERR_SHAPE, "append of %d tokens too large for one call: append it in chunks", L);
  cudaError_t e = ensure_init(cache, (cudaStream_t)stream);
  if (e == cudaSuccess) e = launch_append(cache->g, L, k, v, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "kvq_append_pack launch");
  cache->T += L;
  return KVQ_OK;
}

// ---------------------------------------------------------------------------
// Ragged and paged layouts: per-sequence counts on the host and the device,
// and the page pool's allocator (host side; the device reads the table)
// ---------------------------------------------------------------------------
kvq_status kvq_append_pack_ragged(kvq_cache* cache, const void* k, const void* v, int L,
                                  const int* n, void* stream) {
  if (!cache) return fail(KVQ_ERR_ARG, "cache is NULL");
  const Geom& g = cache->g;
  if (g.layout == KVQ_LAYOUT_UNIFORM)
    return fail(KVQ_ERR_UNSUPPORTED, "kvq_append_pack_ragged needs a ragged or paged cache");
  if (L < 0) return fail(KVQ_ERR_ARG, "L = %d < 0", L);
  std::vector<int> cnt(g.B, L);
  if (n)
    for (int b = 0; b < g.B; ++b) {
      if (n[b] < 0 || n[b] > L) return fail(KVQ_ERR_ARG, "n[%d] = %d outside [0, %d]", b, n[b], L);
      cnt[b] = n[b];
    }
  int total = 0;
  for (int b = 0; b < g.B; ++b) total += cnt[b];
  if (total > 0 && (!k || !v)) return fail(KVQ_ERR_ARG, "k or v is NULL");
  if (misaligned(k) || misaligned(v)) return fail(KVQ_ERR_ARG, "k and v must be 16-byte aligned");
  if ((int64_t)g.B * g.H * (int64_t)L * (g.D / 4) >= ((int64_t)1 << 31))
    return fail(KVQ_ERR_SHAPE, "append of %d tokens too large for one call: append it in chunks", L);
  // capacity, and the pages the new tokens need (taken only if all fit)
  int need_pages = 0;
  for (int b = 0; b < g.B; ++b) {
    const int64_t t1 = (int64_t)cache->seq_T[b] + cnt[b];
    if (t1 > g.Tmax)
      return fail(KVQ_ERR_CAPACITY, "sequence %d: %d + %d tokens exceed max_tokens %d", b,
                  cache->seq_T[b], cnt[b], g.Tmax);
    if (g.layout == KVQ_LAYOUT_PAGED)
      need_pages += (int)((t1 + kPageTok - 1) / kPageTok) - (int)cache->seq_pages[b].size();
  }
  if (need_pages > (int)cache->free_pages.size())
    return fail(KVQ_ERR_CAPACITY, "the append needs %d pages, %d are free", need_pages,
                (int)cache->free_pages.size());
  cudaStream_t s = (cudaStream_t)stream;
  cudaError_t e = ensure_init(cache, s);
  if (e != cudaSuccess) return cuda_fail(e, "kvq_append_pack_ragged");
  if (g.layout == KVQ_LAYOUT_PAGED) {
    for (int b = 0; b < g.B; ++b) {
      std::vector<int>& pg = cache->seq_pages[b];
      const int have = (int)pg.size();
      const int want = (cache->seq_T[b] + cnt[b] + kPageTok - 1) / kPageTok;
      if (want <= have) continue;
      for (int i = have; i < want; ++i) {
        pg.push_back(cache->free_pages.back());
        cache->free_pages.pop_back();
      }
      // the table entries travel with the stream (a pageable copy is staged
      // before the call returns, so pg may change afterwards)
      e = cudaMemcpyAsync(g.page_table + (size_t)b * g.max_pages + have, pg.data() + have,
                          (size_t)(want - have) * sizeof(int32_t), cudaMemcpyHostToDevice, s);
      if (e != cudaSuccess) return cuda_fail(e, "kvq_append_pack_ragged page table");
    }
  }
  e = launch_append_ragged(g, L, k, v, cnt.data(), s);
  if (e != cudaSuccess) return cuda_fail(e, "kvq_append_pack_ragged launch");
  int tmax = 0;
  for (int b = 0; b < g.B; ++b) {
    cache->seq_T[b] += cnt[b];
    cache->seq_n[b] = cnt[b];
    tmax = std::max(tmax, cache->seq_T[b]);
  }
  cache->T = tmax;
  return KVQ_OK;
}

int kvq_seq_tokens(const kvq_cache* cache, int b) {
  if (!cache || b < 0 || b >= cache->g.B) return -1;
  return cache->g.layout == KVQ_LAYOUT_UNIFORM ? cache->T : cache->seq_T[b];
}

kvq_status kvq_seq_release(kvq_cache* cache, int b, void* stream) {
  if (!cache) return fail(KVQ_ERR_ARG, "cache is NULL");
  if (cache->g.layout == KVQ_LAYOUT_UNIFORM)
    return fail(KVQ_ERR_UNSUPPORTED, "kvq_seq_release needs a ragged or paged cache");
  if (b < 0 || b >= cache->g.B) return fail(KVQ_ERR_ARG, "sequence %d outside [0, %d)", b, cache->g.B);
  cudaStream_t s = (cudaStream_t)stream;
  cudaError_t e = ensure_init(cache, s);
  if (e == cudaSuccess) e = launch_seq_reset(cache->g, b, s);
  if (e != cudaSuccess) return cuda_fail(e, "kvq_seq_release");
  for (int p : cache->seq_pages[b]) cache->free_pages.push_back(p);
  cache->seq_pages[b].clear();
  cache->seq_T[b] = cache->seq_n[b] = 0;
  int tmax = 0;
  for (int x : cache->seq_T) tmax = std::max(tmax, x);
  cache->T = tmax;
  return KVQ_OK;
}

int kvq_free_pages(const kvq_cache* cache) {
  if (!cache || cache->g.layout != KVQ_LAYOUT_PAGED) return -1;
  return (int)cache->free_pages.size();
}

int kvq_seq_pages(const kvq_cache* cache, int b, int* pages, int max_pages) {
  if (!cache || cache->g.layout != KVQ_LAYOUT_PAGED || b < 0 || b >= cache->g.B) return -1;
  const std::vector<int>& pg = cache->seq_pages[b];
  for (int i = 0; i < (int)pg.size() && i < max_pages && pages; ++i) pages[i] = pg[i];
  return (int)pg.size();
}

static kvq_status attend_common(kvq_cache* cache, const void* q, int L, int n_q_heads,
                                float scale, void* out, void* stream, bool decode) {
  if (!cache) return fail(KVQ_ERR_ARG, "cache is NULL");
  if (!q || !out) return fail(KVQ_ERR_ARG, "q or out is NULL");
  if (misaligned(q) || misaligned(out)) return fail(KVQ_ERR_ARG, "q and out must be 16-byte aligned");
  if (L <= 0) return fail(KVQ_ERR_ARG, "L = %d must be positive", L);
  if (n_q_heads != cache->g.Hq)
    return fail(KVQ_ERR_SHAPE, "n_q_heads %d != cache q_heads %d", n_q_heads, cache->g.Hq);
  if (cache->g.layout == KVQ_LAYOUT_UNIFORM && L > cache->T)
    return fail(KVQ_ERR_SHAPE, "%d queries but only %d cached tokens (append first)", L,
                cache->T);
  if (cache->g.layout != KVQ_LAYOUT_UNIFORM && !decode)
    for (int b = 0; b < cache->g.B; ++b)
      if (cache->seq_n[b] > L)
        return fail(KVQ_ERR_SHAPE, "sequence %d appended %d tokens, more than L = %d query rows",
                    b, cache->seq_n[b], L);
  if (!(scale > 0.f) || scale != scale) return fail(KVQ_ERR_ARG, "softmax_scale must be > 0");
  if (cache->g.layout != KVQ_LAYOUT_UNIFORM) {
    // a streaming decode over N blocks in P equal ranges gives a head of m
    // blocks at most ceil(m P / N) + 1 CTAs: P <= 30 N / m keeps that <= 31
    int64_t n = 0, m = 0;
    for (int t : cache->seq_T) {
      n += (int64_t)cache->g.H * ((t + 31) / 32);
      m = std::max<int64_t>(m, (t + 31) / 32);
    }
    cache->g.ragged_cta_cap = m > 0 ? (int)std::max<int64_t>(1, std::min<int64_t>(1 << 20, 30 * n / m)) : 0;
  }
  cudaError_t e = ensure_init(cache, (cudaStream_t)stream);
  if (e == cudaSuccess) e = launch_attend(cache->g, q, L, scale, out, decode, cache->T,
                                            (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "kvq_attend launch");
  return KVQ_OK;
}

kvq_status kvq_attend_prefill(kvq_cache* cache, const void* q, int L, int n_q_heads,
                              float softmax_scale, void* out, void* stream) {
  return attend_common(cache, q, L, n_q_heads, softmax_scale, out, stream, false);
}

kvq_status kvq_attend_decode(kvq_cache* cache, const void* q, int n_q_heads,
                             float softmax_scale, void* out, void* stream) {
  return attend_common(cache, q, 1, n_q_heads, softmax_scale, out, stream, true);
}

kvq_status kvq_project_lora(const void* x, int B, int L, int d_in, const void* w_qkv,
                            const void* a_q, const void* b_q, int r_q,
                            const void* a_k, const void* b_k, int r_k,
                            const void* a_v, const void* b_v, int r_v,
                            float alpha_over_r, int n_q_heads, int n_kv_heads,
                            int head_dim, int pos0, kvq_cache* pos_cache, float rope_base,
                            int dtype, void* q, void* k, void* v, void* stream) {
  if (dtype != KVQ_F32 && dtype != KVQ_BF16) return fail(KVQ_ERR_ARG, "unknown dtype %d", dtype);
  if (B < 0 || L < 0 || d_in <= 0) return fail(KVQ_ERR_SHAPE, "bad B/L/d_in");
  if (n_q_heads <= 0 || n_kv_heads <= 0 || n_q_heads % n_kv_heads)
    return fail(KVQ_ERR_SHAPE, "heads %d/%d", n_q_heads, n_kv_heads);
  if (head_dim != 64 && head_dim != 128 && head_dim != 256)
    return fail(KVQ_ERR_UNSUPPORTED, "head_dim %d (supported: 64, 128, 256)", head_dim);
  if (pos0 < 0) return fail(KVQ_ERR_ARG, "pos0 < 0");
  if (!(rope_base >= 0.f)) return fail(KVQ_ERR_ARG, "rope_base < 0");
  if (dtype == KVQ_BF16 && d_in % 64 != 0)
    return fail(KVQ_ERR_SHAPE, "d_in %d must be a multiple of 64 for bf16", d_in);
  if (B == 0 || L == 0) return KVQ_OK;
  if (!x || !w_qkv || !q || !k || !v) return fail(KVQ_ERR_ARG, "NULL tensor pointer");
  if (misaligned(x) || misaligned(w_qkv) || misaligned(q) || misaligned(k) || misaligned(v))
    return fail(KVQ_ERR_ARG, "tensor pointers must be 16-byte aligned");
  const void* a[3] = {a_q, a_k, a_v};
  const void* bm[3] = {b_q, b_k, b_v};
  int r[3] = {r_q, r_k, r_v};
  for (int p = 0; p < 3; ++p) {
    if (r[p] < 0 || r[p] > 64) return fail(KVQ_ERR_SHAPE, "rank %d outside [0, 64]", r[p]);
    if (r[p] > 0 && (!a[p] || !bm[p])) return fail(KVQ_ERR_ARG, "rank %d but NULL factor", r[p]);
    if (dtype == KVQ_BF16 && r[p] % 8) return fail(KVQ_ERR_SHAPE, "bf16 rank %d not a multiple of 8", r[p]);
    if (r[p] == 0) { a[p] = nullptr; bm[p] = nullptr; }
    if (misaligned(a[p]) || misaligned(bm[p]))
      return fail(KVQ_ERR_ARG, "LoRA factors must be 16-byte aligned");
  }
  void* out[3] = {q, k, v};
  int* err = device_error_word();
  if (!err) return fail(KVQ_ERR_CUDA, "cannot resolve the device error word");
  const int* pos_dev = nullptr;
  int pos_stride = 0;
  if (pos_cache) {
    cudaError_t e0 = ensure_init(pos_cache, (cudaStream_t)stream);
    if (e0 != cudaSuccess) return cuda_fail(e0, "kvq_project_lora");
    if (pos_cache->g.layout != KVQ_LAYOUT_UNIFORM) {   // each sequence at its own count
      if (B > pos_cache->g.B) return fail(KVQ_ERR_SHAPE, "B %d > the cache's %d sequences", B, pos_cache->g.B);
      pos_dev = pos_cache->g.seq_len;
      pos_stride = 1;
    } else {
      pos_dev = &pos_cache->g.state->tokens;
    }
  }
  cudaError_t e = launch_project(x, B, L, d_in, w_qkv, a, bm, r, alpha_over_r, n_q_heads,
                                 n_kv_heads, head_dim, pos0, pos_dev, rope_base, dtype, out,
                                 err, (cudaStream_t)stream, pos_stride);
  if (e != cudaSuccess) return cuda_fail(e, "kvq_project_lora launch");
  return KVQ_OK;
}

kvq_status kvq_project_lora_nf4(const void* x, int B, int L, int d_in, const void* w_codes,
                                const void* w_absmax, const void* a_q, const void* b_q, int r_q,
                                const void* a_k, const void* b_k, int r_k,
                                const void* a_v, const void* b_v, int r_v,
                                float alpha_over_r, int n_q_heads, int n_kv_heads, int head_dim,
                                int pos0, kvq_cache* pos_cache, float rope_base, void* q, void* k,
                                void* v, void* stream) {
  if (B < 0 || L < 0 || d_in <= 0) return fail(KVQ_ERR_SHAPE, "bad B/L/d_in");
  if (n_q_heads <= 0 || n_kv_heads <= 0 || n_q_heads % n_kv_heads)
    return fail(KVQ_ERR_SHAPE, "heads %d/%d", n_q_heads, n_kv_heads);
  if (pos0 < 0) return fail(KVQ_ERR_ARG, "pos0 < 0");
  if (!(rope_base >= 0.f)) return fail(KVQ_ERR_ARG, "rope_base < 0");
  const int r[3] = {r_q, r_k, r_v};
  if (!project_nf4_supported(d_in, n_q_heads, n_kv_heads, head_dim, r))
    return fail(KVQ_ERR_UNSUPPORTED,
                "NF4 projection: needs d_in %% 64 == 0, head_dim 64 or 128, Hq*D and Hkv*D "
                "multiples of 128, ranks multiples of 8 up to 64");
  if (B == 0 || L == 0) return KVQ_OK;
  if (!x || !w_codes || !w_absmax || !q || !k || !v) return fail(KVQ_ERR_ARG, "NULL tensor pointer");
  if (misaligned(x) || misaligned(w_codes) || misaligned(q) || misaligned(k) || misaligned(v) ||
      (reinterpret_cast<uintptr_t>(w_absmax) & 3))
    return fail(KVQ_ERR_ARG, "tensor pointers must be 16-byte aligned (absmax: 4-byte)");
  const void* a[3] = {a_q, a_k, a_v};
  const void* bm[3] = {b_q, b_k, b_v};
  for (int p = 0; p < 3; ++p) {
    if (r[p] > 0 && (!a[p] || !bm[p])) return fail(KVQ_ERR_ARG, "rank %d but NULL factor", r[p]);
    if (r[p] == 0) { a[p] = nullptr; bm[p] = nullptr; }
    if (misaligned(a[p]) || misaligned(bm[p]))
      return fail(KVQ_ERR_ARG, "LoRA factors must be 16-byte aligned");
  }
  const int* pos_dev = nullptr;
  int pos_stride = 0;
  if (pos_cache) {
    cudaError_t e0 = ensure_init(pos_cache, (cudaStream_t)stream);
    if (e0 != cudaSuccess) return cuda_fail(e0, "kvq_project_lora_nf4");
    if (pos_cache->g.layout != KVQ_LAYOUT_UNIFORM) {   // each sequence at its own count
      if (B > pos_cache->g.B) return fail(KVQ_ERR_SHAPE, "B %d > the cache's %d sequences", B, pos_cache->g.B);
      pos_dev = pos_cache->g.seq_len;
      pos_stride = 1;
    } else {
      pos_dev = &pos_cache->g.state->tokens;
    }
  }
  void* out[3] = {q, k, v};
  cudaError_t e;
  if (B * L > 16 && project_tc_nf4_supported(n_q_heads, n_kv_heads, head_dim, d_in)) {
    // prefill rows: tcgen05, the base dequantised in the kernel's operand path
    int* err = device_error_word();
    if (!err) return cuda_fail(cudaErrorInvalidDevice, "kvq_project_lora_nf4");
    e = launch_project_tc_nf4(x, B, L, d_in, w_codes, w_absmax, a, bm, r, alpha_over_r,
                              n_q_heads, n_kv_heads, head_dim, pos0, pos_dev, rope_base, out, err,
                              (cudaStream_t)stream, pos_stride);
  } else {
    e = launch_project_nf4(x, B, L, d_in, w_codes, w_absmax, a, bm, r, alpha_over_r, n_q_heads,
                           n_kv_heads, head_dim, pos0, pos_dev, rope_base, out,
                           (cudaStream_t)stream, pos_stride);
  }
  if (e != cudaSuccess) return cuda_fail(e, "kvq_project_lora_nf4 launch");
  return KVQ_OK;
}

// The shapes the fused projection-and-append covers (no launch).
static const char* project_append_gap(const kvq_cache* c, int L, int d_in, const int r[3]) {
  const Geom& g = c->g;
  if (g.layout != KVQ_LAYOUT_UNIFORM) return "the cache is ragged or paged";
  if (g.act != KVQ_BF16) return "the activation dtype is not bf16";
  if (g.fmt != KVQ_FMT_AFFINE && g.fmt != KVQ_FMT_SYMMETRIC) return "the cache is not affine or symmetric";
  if (g.G != 32) return "the group size is not 32";
  for (int b : {g.kb, g.vb})
    if (b != 2 && b != 4 && b != 8) return "code widths must be 2, 4 or 8 bits";
  if ((int64_t)g.B * L <= 16) return "16 rows or fewer (decode rows take the weight-streaming kernel)";
  if (d_in <= 0 || d_in % 64) return "d_in is not a positive multiple of 64";
  if (!project_tc_tile(g.Hq, g.H, g.D, d_in)) return "the head shapes do not tile the tensor-core kernel";
  for (int p = 0; p < 3; ++p)
    if (r[p] < 0 || r[p] > 64 || r[p] % 8) return "LoRA ranks must be multiples of 8 up to 64";
  return nullptr;
}

int kvq_project_append_supported(const kvq_cache* cache, int L, int d_in, int r_q, int r_k,
                                 int r_v) {
  if (!cache) return -1;
  const int r[3] = {r_q, r_k, r_v};
  return project_append_gap(cache, L, d_in, r) == nullptr ? 1 : 0;
}

kvq_status kvq_project_append(kvq_cache* cache, const void* x, int L, int d_in,
                              const void* w_qkv, const void* a_q, const void* b_q, int r_q,
                              const void* a_k, const void* b_k, int r_k,
                              const void* a_v, const void* b_v, int r_v,
                              float alpha_over_r, float rope_base, void* q, void* stream) {
  if (!cache) return fail(KVQ_ERR_ARG, "cache is NULL");
  if (L < 0) return fail(KVQ_ERR_ARG, "L = %d < 0", L);
  if (!(rope_base >= 0.f)) return fail(KVQ_ERR_ARG, "rope_base < 0");
  if (L == 0) return KVQ_OK;
  const Geom& g = cache->g;
  const int r[3] = {r_q, r_k, r_v};
  if (const char* why = project_append_gap(cache, L, d_in, r))
    return fail(KVQ_ERR_UNSUPPORTED, "kvq_project_append: %s", why);
  if (!x || !w_qkv || !q) return fail(KVQ_ERR_ARG, "NULL tensor pointer");
  if (misaligned(x) || misaligned(w_qkv) || misaligned(q))
    return fail(KVQ_ERR_ARG, "tensor pointers must be 16-byte aligned");
  const void* a[3] = {a_q, a_k, a_v};
  const void* bm[3] = {b_q, b_k, b_v};
  for (int p = 0; p < 3; ++p) {
    if (r[p] > 0 && (!a[p] || !bm[p])) return fail(KVQ_ERR_ARG, "rank %d but NULL factor", r[p]);
    if (r[p] == 0) { a[p] = nullptr; bm[p] = nullptr; }
    if (misaligned(a[p]) || misaligned(bm[p]))
      return fail(KVQ_ERR_ARG, "LoRA factors must be 16-byte aligned");
  }
  if ((int64_t)cache->T + L > g.Tmax)
    return fail(KVQ_ERR_CAPACITY, "append of %d tokens to %d exceeds max_tokens %d", L, cache->T,
                g.Tmax);
  int* err = device_error_word();
  if (!err) return fail(KVQ_ERR_CUDA, "cannot resolve the device error word");
  cudaError_t e = ensure_init(cache, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "kvq_project_append");
  void* out[3] = {q, nullptr, nullptr};
  e = launch_project_tc(x, g.B, L, d_in, w_qkv, a, bm, r, alpha_over_r, g.Hq, g.H, g.D, 0,
                        &cache->g.state->tokens, rope_base, out, err, (cudaStream_t)stream, &g);
  if (e != cudaSuccess) return cuda_fail(e, "kvq_project_append launch");
  cache->T += L;
  return KVQ_OK;
}

kvq_status kvq_decode_step(kvq_cache* cache, const void* x, int d_in, const void* w_qkv,
                           const void* a_q, const void* b_q, int r_q,
                           const void* a_k, const void* b_k, int r_k,
                           const void* a_v, const void* b_v, int r_v,
                           float alpha_over_r, float rope_base, float softmax_scale,
                           void* q, void* k, void* v, void* out, void* stream) {
  if (!cache) return fail(KVQ_ERR_ARG, "cache is NULL");
  const Geom& g = cache->g;
  if (!out) return fail(KVQ_ERR_ARG, "out is NULL");
  if (misaligned(out)) return fail(KVQ_ERR_ARG, "out must be 16-byte aligned");
  if (!(softmax_scale > 0.f)) return fail(KVQ_ERR_ARG, "softmax_scale must be > 0");
  if (cache->T + 1 > g.Tmax)
    return fail(KVQ_ERR_CAPACITY, "decode step on a full cache (%d tokens)", cache->T);
  const int r[3] = {r_q, r_k, r_v};
  const void* a[3] = {a_q, a_k, a_v};
  const void* bm[3] = {b_q, b_k, b_v};
  if (g.act == KVQ_BF16 && decode_step_supported(g, d_in, r)) {
    // same validation as the separate calls
    kvq_status st = KVQ_OK;
    if (d_in <= 0 || d_in % 64) st = fail(KVQ_ERR_SHAPE, "d_in %d must be a multiple of 64", d_in);
    if (!x || !w_qkv || !q || !k || !v) st = fail(KVQ_ERR_ARG, "NULL tensor pointer");
    if (st == KVQ_OK && (misaligned(x) || misaligned(w_qkv) || misaligned(q) || misaligned(k) ||
                         misaligned(v)))
      st = fail(KVQ_ERR_ARG, "tensor pointers must be 16-byte aligned");
    for (int p = 0; p < 3 && st == KVQ_OK; ++p) {
      if (r[p] < 0 || r[p] % 8) st = fail(KVQ_ERR_SHAPE, "bf16 rank %d not a multiple of 8", r[p]);
      else if (r[p] > 0 && (!a[p] || !bm[p])) st = fail(KVQ_ERR_ARG, "rank %d but NULL factor", r[p]);
      else if (r[p] > 0 && (misaligned(a[p]) || misaligned(bm[p])))
        st = fail(KVQ_ERR_ARG, "LoRA factors must be 16-byte aligned");
    }
    if (st != KVQ_OK) return st;
    const void* aa[3] = {r_q ? a_q : nullptr, r_k ? a_k : nullptr, r_v ? a_v : nullptr};
    const void* bb[3] = {r_q ? b_q : nullptr, r_k ? b_k : nullptr, r_v ? b_v : nullptr};
    int* err = device_error_word();
    if (!err) return fail(KVQ_ERR_CUDA, "cannot resolve the device error word");
    cudaStream_t s = (cudaStream_t)stream;
    cudaError_t e = ensure_init(cache, s);
    void* qkv[3] = {q, k, v};
    if (e == cudaSuccess)
      e = launch_decode_step(g, x, d_in, w_qkv, aa, bb, r, alpha_over_r, rope_base, softmax_scale,
                             qkv, out, err, s);
    if (e != cudaErrorNotSupported) {
      if (e != cudaSuccess) return cuda_fail(e, "kvq_decode_step launch");
      cache->T += 1;
      return KVQ_OK;
    }
    (void)cudaGetLastError();
  }
  // general path: the three calls in sequence
  kvq_status st = kvq_project_lora(x, g.B, 1, d_in, w_qkv, a_q, b_q, r_q, a_k, b_k, r_k, a_v, b_v,
                                   r_v, alpha_over_r, g.Hq, g.H, g.D, 0, cache, rope_base, g.act,
                                   q, k, v, stream);
  if (st == KVQ_OK) st = kvq_append_pack(cache, k, v, 1, stream);
  if (st == KVQ_OK) st = kvq_attend_decode(cache, q, g.Hq, softmax_scale, out, stream);
  return st;
}

int kvq_decode_step_fused(const kvq_cache* cache, int d_in, int r_q, int r_k, int r_v) {
  if (!cache) return -1;
  const int r[3] = {r_q, r_k, r_v};
  return cache->g.act == KVQ_BF16 && decode_step_supported(cache->g, d_in, r) ? 1 : 0;
}

static const char* attend_backward_gap(const kvq_cache* c, int L, int n_q_heads) {
  if (c->g.fmt == KVQ_FMT_KVARN) return "KVarN caches have no backward";
  if (c->g.layout != KVQ_LAYOUT_UNIFORM) return "ragged and paged caches have no backward";
  if (L <= 0) return "L must be positive";
  if (n_q_heads != c->g.Hq) return "n_q_heads differs from the cache's q_heads";
  if (L > c->T) return "more queries than cached tokens (append first)";
  return nullptr;
}

size_t kvq_attend_backward_workspace(const kvq_cache* cache, int L, int n_q_heads) {
  if (!cache || attend_backward_gap(cache, L, n_q_heads)) return 0;
  return attend_backward_pair_bytes(cache->g, cache->T, L);
}

kvq_status kvq_attend_backward(kvq_cache* cache, const void* q, const void* d_out, int L,
                               int n_q_heads, float softmax_scale, float* d_q, float* d_k,
                               float* d_v, void* workspace, size_t workspace_bytes,
                               void* stream) {
  if (!cache) return fail(KVQ_ERR_ARG, "cache is NULL");
  if (const char* gap = attend_backward_gap(cache, L, n_q_heads))
    return fail(cache->g.fmt == KVQ_FMT_KVARN || cache->g.layout != KVQ_LAYOUT_UNIFORM
                    ? KVQ_ERR_UNSUPPORTED : KVQ_ERR_SHAPE,
                "kvq_attend_backward: %s", gap);
  if (!q || !d_out || !d_q || !d_k || !d_v || !workspace)
    return fail(KVQ_ERR_ARG, "NULL tensor pointer");
  if (misaligned(q) || misaligned(d_out) || misaligned(d_q) || misaligned(d_k) ||
      misaligned(d_v) || misaligned(workspace))
    return fail(KVQ_ERR_ARG, "tensor pointers must be 16-byte aligned");
  if (!(softmax_scale > 0.f)) return fail(KVQ_ERR_ARG, "softmax_scale must be > 0");
  const size_t per = attend_backward_pair_bytes(cache->g, cache->T, L);
  if (workspace_bytes < per)
    return fail(KVQ_ERR_CAPACITY, "workspace of %zu bytes < %zu (one sequence and kv head)",
                workspace_bytes, per);
  cudaError_t e = ensure_init(cache, (cudaStream_t)stream);
  if (e == cudaSuccess)
    e = launch_attend_backward(cache->g, cache->T, q, d_out, L, softmax_scale, d_q, d_k, d_v,
                               workspace, workspace_bytes, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "kvq_attend_backward launch");
  return KVQ_OK;
}

size_t kvq_lora_backward_workspace(int B, int L, int d_in, int n_q_heads, int n_kv_heads,
                                   int head_dim, int r_q, int r_k, int r_v) {
  if (B <= 0 || L <= 0 || d_in <= 0 || n_q_heads <= 0 || n_kv_heads <= 0 || head_dim <= 0 ||
      r_q < 0 || r_k < 0 || r_v < 0)
    return 0;
  const int r[3] = {r_q, r_k, r_v};
  return lora_backward_bytes(B, L, d_in, n_q_heads, n_kv_heads, head_dim, r);
}

kvq_status kvq_lora_backward(const void* x, int B, int L, int d_in, const void* w_qkv,
                             const void* a_q, const void* b_q, int r_q,
                             const void* a_k, const void* b_k, int r_k,
                             const void* a_v, const void* b_v, int r_v,
                             float alpha_over_r, int n_q_heads, int n_kv_heads, int head_dim,
                             int pos0, float rope_base, int dtype,
                             const float* d_q, const float* d_k, const float* d_v, int kv_rows,
                             float* da_q, float* db_q, float* da_k, float* db_k,
                             float* da_v, float* db_v, float* d_x,
                             void* workspace, size_t workspace_bytes, void* stream) {
  if (dtype != KVQ_F32 && dtype != KVQ_BF16) return fail(KVQ_ERR_ARG, "unknown dtype %d", dtype);
  if (B <= 0 || L <= 0 || d_in <= 0) return fail(KVQ_ERR_SHAPE, "bad B/L/d_in");
  if (n_q_heads <= 0 || n_kv_heads <= 0 || n_q_heads % n_kv_heads)
    return fail(KVQ_ERR_SHAPE, "heads %d/%d", n_q_heads, n_kv_heads);
  if (head_dim != 64 && head_dim != 128 && head_dim != 256)
    return fail(KVQ_ERR_UNSUPPORTED, "head_dim %d (supported: 64, 128, 256)", head_dim);
  if (pos0 < 0 || !(rope_base >= 0.f)) return fail(KVQ_ERR_ARG, "pos0 < 0 or rope_base < 0");
  if (kv_rows < L) return fail(KVQ_ERR_SHAPE, "kv_rows %d < L %d", kv_rows, L);
  if (!x || !d_q || !d_k || !d_v || !workspace) return fail(KVQ_ERR_ARG, "NULL tensor pointer");
  if (d_x && !w_qkv) return fail(KVQ_ERR_ARG, "d_x needs w_qkv");
  const void* a[3] = {a_q, a_k, a_v};
  const void* bm[3] = {b_q, b_k, b_v};
  float* da[3] = {da_q, da_k, da_v};
  float* db[3] = {db_q, db_k, db_v};
  const int r[3] = {r_q, r_k, r_v};
  for (int p = 0; p < 3; ++p) {
    if (r[p] < 0 || r[p] > 64) return fail(KVQ_ERR_SHAPE, "rank %d outside [0, 64]", r[p]);
    if (r[p] > 0 && (!a[p] || !bm[p] || !da[p] || !db[p]))
      return fail(KVQ_ERR_ARG, "rank %d but a NULL factor or gradient", r[p]);
  }
  const size_t need = lora_backward_bytes(B, L, d_in, n_q_heads, n_kv_heads, head_dim, r);
  if (workspace_bytes < need)
    return fail(KVQ_ERR_CAPACITY, "workspace of %zu bytes < %zu", workspace_bytes, need);
  if (misaligned(workspace)) return fail(KVQ_ERR_ARG, "workspace must be 16-byte aligned");
  cudaError_t e = launch_lora_backward(x, B, L, d_in, w_qkv, a, bm, r, alpha_over_r, n_q_heads,
                                       n_kv_heads, head_dim, pos0, rope_base, dtype, d_q, d_k,
                                       d_v, kv_rows, da, db, d_x, workspace, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "kvq_lora_backward launch");
  return KVQ_OK;
}

kvq_status kvq_device_status(void* stream, int* out) {
  if (!out) return fail(KVQ_ERR_ARG, "out is NULL");
  int* p = device_error_word();
  if (!p) return fail(KVQ_ERR_CUDA, "cannot resolve the device error word");
  cudaStream_t s = (cudaStream_t)stream;
  int h = 0;
  cudaError_t e = cudaMemcpyAsync(&h, p, sizeof(int), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaMemsetAsync(p, 0, sizeof(int), s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(e, "kvq_device_status");
  *out = h;
  return h ? KVQ_ERR_TIMEOUT : KVQ_OK;
}

}  // extern "C"
