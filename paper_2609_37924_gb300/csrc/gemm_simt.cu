// fp32 GEMM on the CUDA cores, used by fp32 models (the tiny workload):
// acc[M, N] = A[M, K] * B[N, K]^T with the same fused epilogues as the tensor
// core path.  64 x 64 output tile per 256-thread block, 4 x 4 per thread,
// K staged through shared memory 16 at a time.  EPI_GLU tiles hold 32 gate
// and 32 up columns; EPI_QKV needs head_dim <= 64.
#include "kernels.h"

namespace tadm {
namespace {
constexpr int TM = 64, TN = 64, TK = 16;

struct SmemSrc {
  static constexpr bool kStaged = false;
  __device__ bool staged() const { return false; }
  __device__ void store64(int, int, const float (&)[32], const float (&)[32]) {}
  const float* row;  // accumulator row in shared memory
  __device__ __forceinline__ void load(int chunk, float (&v)[32]) {
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = row[32 * chunk + i];
  }
};

template <int EPI>
__global__ void __launch_bounds__(256) gemm_simt_kernel(const float* __restrict__ A, const float* __restrict__ B,
                                                        int M, int K, int lda, int ldb, int n_rows_b,
                                                        int b_split, EpiParams ep) {
  pdl_enter();
  __shared__ float sA[TK][TM + 4];
  __shared__ float sB[TK][TN + 4];
  __shared__ float sC[TM][TN + 1];
  const int tid = threadIdx.x;
  const int tx = tid % 16, ty = tid / 16;
  const int m0 = blockIdx.y * TM, nb = blockIdx.x;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < K; k0 += TK) {
    for (int i = tid; i < TM * TK; i += 256) {
      const int r = i / TK, c = i % TK;
      const int gm = m0 + r, gk = k0 + c;
      sA[c][r] = (gm < M && gk < K) ? A[static_cast<size_t>(gm) * lda + gk] : 0.0f;
      int gn;
      if (b_split > 0) gn = (r < TN / 2) ? nb * (TN / 2) + r : b_split + nb * (TN / 2) + (r - TN / 2);
      else gn = nb * TN + r;
      sB[c][r] = (gn < n_rows_b && gk < K) ? B[static_cast<size_t>(gn) * ldb + gk] : 0.0f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < TK; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) { a[i] = sA[kk][ty * 4 + i]; b[i] = sB[kk][tx * 4 + i]; }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) sC[ty * 4 + i][tx * 4 + j] = acc[i][j];
  __syncthreads();
  if (tid < TM) {
    SmemSrc src{&sC[tid][0]};
    epilogue_row<EPI>(ep, m0 + tid, nb, TN, src);
  }
}

template <int EPI>
cudaError_t launch(const GemmCall& g, int tiles_n, int b_split, int n_rows_b, const EpiParams& ep, cudaStream_t s) {
  dim3 grid(tiles_n, (g.M + TM - 1) / TM);
  launch_pdl(gemm_simt_kernel<EPI>, grid, 256, 0, s, static_cast<const float*>(g.A), static_cast<const float*>(g.B), g.M,
                                             g.K, g.lda, g.ldb, n_rows_b, b_split, ep);
  return cudaGetLastError();
}
}  // namespace

int gemm_simt_tiles_n(int N, int epi) { return epi == EPI_GLU ? (N + 31) / 32 : (N + 63) / 64; }

const char* gemm_simt(const GemmCall& g, cudaStream_t s) {
  if (g.M <= 0 || g.N <= 0 || g.K <= 0) return nullptr;
  const bool glu = g.epi == EPI_GLU;
  if (glu && g.N % 32) return "GLU GEMM (fp32) needs the FFN width to be a multiple of 32";
  if (g.epi == EPI_QKV && TN % g.ep.head_dim) return "fp32 path needs head_dim dividing 64";
  if (g.epi == EPI_PA_GATE && g.N > TN) return "fp32 gate GEMM needs N <= 64";
  const int tiles_n = gemm_simt_tiles_n(g.N, g.epi);
  EpiParams ep = g.ep;
  ep.M = g.M;
  ep.N = g.N;
  ep.n_tiles = tiles_n;
  const int b_split = glu ? g.N : 0;
  const int n_rows_b = glu ? 2 * g.N : g.N;
  cudaError_t e;
  switch (g.epi) {
    case EPI_STORE: e = launch<EPI_STORE>(g, tiles_n, b_split, n_rows_b, ep, s); break;
    case EPI_RESID: e = launch<EPI_RESID>(g, tiles_n, b_split, n_rows_b, ep, s); break;
    case EPI_QKV: e = launch<EPI_QKV>(g, tiles_n, b_split, n_rows_b, ep, s); break;
    case EPI_GLU: e = launch<EPI_GLU>(g, tiles_n, b_split, n_rows_b, ep, s); break;
    case EPI_FUSION1: e = launch<EPI_FUSION1>(g, tiles_n, b_split, n_rows_b, ep, s); break;
    case EPI_FUSION2: e = launch<EPI_FUSION2>(g, tiles_n, b_split, n_rows_b, ep, s); break;
    case EPI_LMHEAD: e = launch<EPI_LMHEAD>(g, tiles_n, b_split, n_rows_b, ep, s); break;
    case EPI_PA_UP: e = launch<EPI_PA_UP>(g, tiles_n, b_split, n_rows_b, ep, s); break;
    case EPI_SILU: e = launch<EPI_SILU>(g, tiles_n, b_split, n_rows_b, ep, s); break;
    case EPI_ADD: e = launch<EPI_ADD>(g, tiles_n, b_split, n_rows_b, ep, s); break;
    case EPI_PA_GATE: e = launch<EPI_PA_GATE>(g, tiles_n, b_split, n_rows_b, ep, s); break;
    default: return "unknown epilogue";
  }
  return e == cudaSuccess ? nullptr : cudaGetErrorString(e);
}

}  // namespace tadm
