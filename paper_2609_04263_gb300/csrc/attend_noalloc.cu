// Decode attention for callers that cannot allocate device memory.
//
// kvq_attend_decode keeps its split-K partials in the workspace plane of the
// cache buffer, which the caller sized with kvq_cache_bytes() and allocated.
// Some callers cannot provide that memory at call time: a plugin or custom-op
// host that hands the op only its input and output tensors and forbids
// allocation, code that runs where cudaMalloc would synchronise the device
// or is not permitted (latency-critical serving loops, allocation-free
// runtimes), or a process whose memory pool already reserves all free HBM.
// This variant keeps the partials in a fixed array in static device memory
// instead, so the call itself allocates nothing.
//
// The array has a fixed maximum size (kNoAllocScratchFloats floats, 4 MiB);
// every GPU that loads the library holds it until the process exits.  Calls
// whose partials would not fit are rejected.  All calls share the one array
// and it keeps the last call's contents: the split kernel writes every
// partial row the merge reads (empty splits included), so nothing needs to
// start at zero, but two calls that overlap on the GPU (different streams,
// or different caches used concurrently) race on it.
#include <mutex>

#include "kvq_internal.cuh"

namespace {

constexpr size_t kNoAllocScratchFloats = size_t(1) << 20;   // 4 MiB of fp32

static __device__ __align__(256) float g_decode_scratch[kNoAllocScratchFloats];

std::mutex g_scratch_mu;

// Device address of the scratch array on the current device.  The first call
// on each device looks it up (cudaGetSymbolAddress) with that device current.
float* scratch_address(cudaError_t* err) {
  static float* addr[64] = {nullptr};
  int dev = 0;
  *err = cudaGetDevice(&dev);
  if (*err != cudaSuccess) return nullptr;
  if (dev < 0 || dev >= 64) {
    *err = cudaErrorInvalidDevice;
    return nullptr;
  }
  std::lock_guard<std::mutex> lk(g_scratch_mu);
  if (!addr[dev]) {
    void* p = nullptr;
    *err = cudaGetSymbolAddress(&p, g_decode_scratch);
    if (*err != cudaSuccess) return nullptr;
    addr[dev] = static_cast<float*>(p);
  }
  return addr[dev];
}

}  // namespace

extern "C" kvq_status kvq_attend_decode_noalloc(kvq_cache* cache, const void* q, int n_q_heads,
                                                float softmax_scale, void* out, void* stream) {
  using namespace kvq;
  if (!cache) return set_error(KVQ_ERR_ARG, "cache is NULL");
  if (!q || !out) return set_error(KVQ_ERR_ARG, "q or out is NULL");
  if ((reinterpret_cast<uintptr_t>(q) & 15) || (reinterpret_cast<uintptr_t>(out) & 15))
    return set_error(KVQ_ERR_ARG, "q and out must be 16-byte aligned");
  if (n_q_heads != cache->g.Hq)
    return set_error(KVQ_ERR_SHAPE, "n_q_heads %d != cache q_heads %d", n_q_heads, cache->g.Hq);
  if (cache->T < 1)
    return set_error(KVQ_ERR_SHAPE, "no cached tokens (append first)");
  if (!(softmax_scale > 0.f)) return set_error(KVQ_ERR_ARG, "softmax_scale must be > 0");
  const size_t need = workspace_floats(cache->g);
  if (need > kNoAllocScratchFloats)
    return set_error(KVQ_ERR_CAPACITY,
                     "decode partials need %zu floats (batch %d x q_heads %d x %d splits x "
                     "(head_dim + 2)); the static scratch holds %zu",
                     need, cache->g.B, cache->g.Hq, kMaxSplits, kNoAllocScratchFloats);
  cudaError_t e;
  float* scratch = scratch_address(&e);
  if (!scratch)
    return set_error(KVQ_ERR_CUDA, "static decode scratch: %s", cudaGetErrorString(e));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  e = ensure_cache_init(cache, s);
  if (e != cudaSuccess) return set_error(KVQ_ERR_CUDA, "kvq_attend_decode_noalloc: %s",
                                         cudaGetErrorString(e));
  Geom g = cache->g;                        // same kernels, partials in the static array
  g.pl[KVQ_PLANE_WORKSPACE].p = scratch;
  e = launch_attend(g, q, 1, softmax_scale, out, true, cache->T, s);
  if (e != cudaSuccess) return set_error(KVQ_ERR_CUDA, "kvq_attend_decode_noalloc launch: %s",
                                         cudaGetErrorString(e));
  return KVQ_OK;
}
