// Split-K flash-decode over the packed cache on tensor cores: the standalone
// kernel (one split per CTA).  The device code is in decode_attn.cuh.
#include "decode_attn.cuh"

namespace kvq {
namespace {
using namespace dattn;

template <int D, int BITS, int FMT>
__global__ void __launch_bounds__(kWarps * 32)
attend_decode_mma_kernel(Geom g, const __nv_bfloat16* __restrict__ q, float scale, int* err,
                         __nv_bfloat16* __restrict__ out) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ __align__(128) unsigned char smem[];
  __shared__ uint64_t bars[kStages];
  const int grp = g.Hq / g.H;
  decode_split<D, BITS, FMT, kStages, kWarps>(
      g, q + ((int64_t)blockIdx.z * g.Hq + blockIdx.y * grp) * D, scale, err, out, blockIdx.x,
      g.splits, kMaxSplits, blockIdx.y, blockIdx.z, seq_tokens(g, blockIdx.z), smem, bars, false);
}

template <int D, int BITS, int FMT>
cudaError_t launch_one(const Geom& g, const void* q, float scale, int* err, void* out,
                       cudaStream_t s) {
  using C = Cfg<D, BITS, FMT>;
  const size_t sm = attn_smem_bytes<D, BITS, FMT>();
  auto kern = attend_decode_mma_kernel<D, BITS, FMT>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm);
  if (e != cudaSuccess) return e;
  launch_pdl(kern, dim3(dim3(g.splits, g.H, g.B)), dim3(kWarps * 32), sm, s, 
      g, reinterpret_cast<const __nv_bfloat16*>(q), scale, err,
      reinterpret_cast<__nv_bfloat16*>(out));
  return cudaGetLastError();
}

template <int D, int BITS>
cudaError_t launch_fmt(const Geom& g, const void* q, float scale, int* err, void* out,
                       cudaStream_t s) {
  switch (g.fmt) {
    case KVQ_FMT_AFFINE: return launch_one<D, BITS, KVQ_FMT_AFFINE>(g, q, scale, err, out, s);
    case KVQ_FMT_SYMMETRIC:
      return launch_one<D, BITS, KVQ_FMT_SYMMETRIC>(g, q, scale, err, out, s);
    case KVQ_FMT_KIVI: return launch_one<D, BITS, KVQ_FMT_KIVI>(g, q, scale, err, out, s);
  }
  return cudaErrorNotSupported;
}

}  // namespace

bool decode_mma_supported(const Geom& g) {
  const bool fmt_ok = g.fmt == KVQ_FMT_AFFINE || g.fmt == KVQ_FMT_SYMMETRIC || g.fmt == KVQ_FMT_KIVI;
  return fmt_ok && g.act == KVQ_BF16 && g.G == 32 && g.kb == g.vb && (g.kb == 2 || g.kb == 4) &&
         (g.D == 64 || g.D == 128) && g.Hq / g.H <= 16;
}

cudaError_t launch_decode_mma(const Geom& g, const void* q, float scale, int* err, void* out,
                              cudaStream_t s) {
  if (g.D == 64) return g.kb == 4 ? launch_fmt<64, 4>(g, q, scale, err, out, s)
                                  : launch_fmt<64, 2>(g, q, scale, err, out, s);
  return g.kb == 4 ? launch_fmt<128, 4>(g, q, scale, err, out, s)
                   : launch_fmt<128, 2>(g, q, scale, err, out, s);
}

}  // namespace kvq
