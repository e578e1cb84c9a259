// Internal declarations shared by the kvq translation units: the cache
// geometry passed to kernels by value, plane addressing, small device helpers
// and the host-side launch entry points of each kernel family.
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <stdint.h>

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

// Everything a kernel needs to address a cache.  Passed by value.
struct Geom {
  int32_t fmt, kb, vb, G, R, S, iters;
  int32_t B, H, Hq, D, Tmax, act;
  int32_t ring;          // KIVI: R + G residual slots
  Plane pl[KVQ_NUM_PLANES];
};

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

// Host-side launchers (each defined in the translation unit of its kernels).
// They return cudaGetLastError() of their launches.
cudaError_t launch_append(const Geom& g, int T0, int L, const void* k, const void* v,
                          cudaStream_t s);
cudaError_t launch_attend(const Geom& g, int T, const void* q, int L, float scale,
                          void* out, bool decode, cudaStream_t s);
cudaError_t launch_project(const void* x, int B, int L, int d_in, const void* w,
                           const void* const a[3], const void* const bm[3], const int r[3],
                           float alpha_over_r, int Hq, int Hkv, int D, int pos0,
                           float rope_base, int act, void* const out[3], int* err,
                           cudaStream_t s);

// Number of decode splits the attention launcher uses for a cache state.
int decode_splits(const Geom& g, int T);

// Device address of the library's error word (set up once per device).
int* device_error_word();

int num_sms();

}  // namespace kvq
