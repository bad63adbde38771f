// Split-K reduction for the tcgen05 GEMM: sums the fp32 partials of the K
// slices in slice order (deterministic) into slice 0, then runs the GEMM's own
// epilogue on that sum, one thread per (output row, column group) of a
// 256-column tile; the residual-add and plain-store epilogues do both in one
// element-wise launch.
#include "kernels.h"

namespace tadm {
namespace {

struct PartSrc {
  static constexpr bool kStaged = false;
  const float* row;      // partial row of slice 0 at this tile's first column
  size_t stride;         // between slices
  int splits;
  __device__ __forceinline__ void load(int chunk, float (&v)[32]) {
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = 0.0f;
    for (int ks = 0; ks < splits; ++ks) {
      const float4* p = reinterpret_cast<const float4*>(row + ks * stride + 32 * chunk);
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const float4 t = p[q];
        v[4 * q] += t.x; v[4 * q + 1] += t.y; v[4 * q + 2] += t.z; v[4 * q + 3] += t.w;
      }
    }
  }
};

// Column groups one thread may take without changing the epilogue's result:
// the output head keeps the tensor-core path's two partials per tile, the
// paired-attention gate needs whole rows, GLU pairs gate / up chunks, QKV
// whole heads; the rest is independent per 32-column chunk.
template <int EPI>
__device__ __forceinline__ int reduce_groups(const EpiParams& ep) {
  if constexpr (EPI == EPI_PA_GATE) return 1;
  else if constexpr (EPI == EPI_LMHEAD) return 2;
  else if constexpr (EPI == EPI_GLU) return 4;
  else if constexpr (EPI == EPI_QKV) return 256 / ep.head_dim;
  else return 8;
}

// block: 32 rows x 8 group slots; thread (row, slot) runs group `slot` if it exists
template <int EPI>
__global__ void __launch_bounds__(256) splitk_reduce_kernel(EpiParams ep, const float* __restrict__ part,
                                                            size_t stride, int ldp, int splits) {
  pdl_enter();
  const int m = blockIdx.x * 32 + (threadIdx.x & 31), slot = threadIdx.x >> 5, nb = blockIdx.y;
  const int groups = reduce_groups<EPI>(ep);
  if (m >= ep.M || slot >= groups) return;
  PartSrc src{part + static_cast<size_t>(m) * ldp + nb * 256, stride, splits};
  epilogue_row<EPI>(ep, m, nb, 256, src, slot, groups);
}

// Phase 1: slice 0 <- sum of all slices in slice order, one float4 per thread.
__global__ void __launch_bounds__(256) splitk_sum_kernel(float* __restrict__ part, size_t stride, size_t n4,
                                                         int splits) {
  pdl_enter();
  const size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x;
  if (i >= n4) return;
  float4* p = reinterpret_cast<float4*>(part);
  float4 a = p[i];
  for (int ks = 1; ks < splits; ++ks) {
    const float4 t = p[i + ks * (stride / 4)];
    a.x += t.x; a.y += t.y; a.z += t.z; a.w += t.w;
  }
  p[i] = a;
}

// Element-wise epilogues (residual add, plain store) in one launch: each
// thread sums four consecutive columns of one row over the slices in slice
// order, then adds them into the residual stream (+ bias) or stores them,
// with coalesced 16-byte accesses.  Same sums in the same order as the
// two-phase path below, so the result does not depend on which one ran.
template <int EPI>
__global__ void __launch_bounds__(256) splitk_elem_kernel(EpiParams ep, const float* __restrict__ part, size_t stride,
                                                          int ldp, int splits) {
  pdl_enter();
  const int n4 = ep.N / 4;
  const size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x;
  if (i >= static_cast<size_t>(ep.M) * n4) return;
  const int m = static_cast<int>(i / n4), n = static_cast<int>(i % n4) * 4;
  const float* p = part + static_cast<size_t>(m) * ldp + n;
  float4 a = *reinterpret_cast<const float4*>(p);
  for (int ks = 1; ks < splits; ++ks) {
    const float4 t = *reinterpret_cast<const float4*>(p + ks * stride);
    a.x += t.x; a.y += t.y; a.z += t.z; a.w += t.w;
  }
  if constexpr (EPI == EPI_RESID) {
    float4* r = reinterpret_cast<float4*>(ep.resid + static_cast<size_t>(m) * ep.ldr + n);
    float4 x = *r;
    if (ep.bias) {
      a.x += ld_param(ep.bias, ep.bias_bf16, n + 0);
      a.y += ld_param(ep.bias, ep.bias_bf16, n + 1);
      a.z += ld_param(ep.bias, ep.bias_bf16, n + 2);
      a.w += ld_param(ep.bias, ep.bias_bf16, n + 3);
    }
    x.x += a.x; x.y += a.y; x.z += a.z; x.w += a.w;
    *r = x;
  } else if (ep.out_bf16) {
    __nv_bfloat162* o = reinterpret_cast<__nv_bfloat162*>(static_cast<bf16*>(ep.out) + static_cast<size_t>(m) * ep.ldo + n);
    o[0] = __floats2bfloat162_rn(a.x, a.y);
    o[1] = __floats2bfloat162_rn(a.z, a.w);
  } else {
    *reinterpret_cast<float4*>(static_cast<float*>(ep.out) + static_cast<size_t>(m) * ep.ldo + n) = a;
  }
}

// true when the element-wise kernel serves this epilogue (aligned rows, N % 4 == 0)
bool elem_ok(int epi, const EpiParams& ep, int ldp) {
  if (ep.N % 4 || ldp % 4) return false;
  if (epi == EPI_RESID)
    return ep.ldr % 4 == 0 && (reinterpret_cast<uintptr_t>(ep.resid) & 15) == 0;
  if (epi == EPI_STORE)
    return ep.ldo % 4 == 0 && (reinterpret_cast<uintptr_t>(ep.out) & 15) == 0;
  return false;
}

// Phase 2: the epilogue on slice 0.
template <int EPI>
cudaError_t launch(const EpiParams& ep, const float* part, size_t stride, int ldp, int splits, int n_tiles_n,
                   cudaStream_t s, int* launches) {
  if constexpr (EPI == EPI_RESID || EPI == EPI_STORE) {
    if (elem_ok(EPI, ep, ldp)) {
      *launches = 1;
      const size_t n = static_cast<size_t>(ep.M) * (ep.N / 4);
      launch_pdl(splitk_elem_kernel<EPI>, static_cast<unsigned>((n + 255) / 256), 256, 0, s, ep, part, stride, ldp,
                 splits);
      return cudaGetLastError();
    }
  }
  *launches = 2;
  const size_t n4 = static_cast<size_t>(ep.M) * ldp / 4;
  launch_pdl(splitk_sum_kernel, static_cast<unsigned>((n4 + 255) / 256), 256, 0, s, const_cast<float*>(part), stride, n4,
                                                                            splits);
  dim3 grid((ep.M + 31) / 32, n_tiles_n);
  launch_pdl(splitk_reduce_kernel<EPI>, grid, 256, 0, s, ep, part, stride, ldp, 1);
  return cudaGetLastError();
}
}  // namespace

const char* splitk_reduce(int epi, const EpiParams& ep, const float* part, size_t stride, int ldp, int splits,
                          int n_tiles_n, cudaStream_t s, int* launches) {
  cudaError_t e;
  switch (epi) {
    case EPI_STORE: e = launch<EPI_STORE>(ep, part, stride, ldp, splits, n_tiles_n, s, launches); break;
    case EPI_RESID: e = launch<EPI_RESID>(ep, part, stride, ldp, splits, n_tiles_n, s, launches); break;
    case EPI_QKV: e = launch<EPI_QKV>(ep, part, stride, ldp, splits, n_tiles_n, s, launches); break;
    case EPI_GLU: e = launch<EPI_GLU>(ep, part, stride, ldp, splits, n_tiles_n, s, launches); break;
    case EPI_FUSION1: e = launch<EPI_FUSION1>(ep, part, stride, ldp, splits, n_tiles_n, s, launches); break;
    case EPI_FUSION2: e = launch<EPI_FUSION2>(ep, part, stride, ldp, splits, n_tiles_n, s, launches); break;
    case EPI_LMHEAD: e = launch<EPI_LMHEAD>(ep, part, stride, ldp, splits, n_tiles_n, s, launches); break;
    case EPI_PA_UP: e = launch<EPI_PA_UP>(ep, part, stride, ldp, splits, n_tiles_n, s, launches); break;
    case EPI_SILU: e = launch<EPI_SILU>(ep, part, stride, ldp, splits, n_tiles_n, s, launches); break;
    case EPI_ADD: e = launch<EPI_ADD>(ep, part, stride, ldp, splits, n_tiles_n, s, launches); break;
    case EPI_PA_GATE: e = launch<EPI_PA_GATE>(ep, part, stride, ldp, splits, n_tiles_n, s, launches); break;
    default: return "unknown epilogue";
  }
  return e == cudaSuccess ? nullptr : cudaGetErrorString(e);
}

}  // namespace tadm
