// The sampler P: logits -> (confidence, token) per position, then the
// deterministic top-k unmask of the active block.
//
//  - zero-masking: the MASK id never wins the argmax (App. B.1.1);
//  - conf = p(tok) = 1 / sum_v exp(l_v - l_tok) over v != MASK;
//  - argmax ties go to the lowest id; selection ties to the lowest position;
//  - carry-over: only positions still holding MASK are candidates, so
//    unmasked tokens never change.
#include "kernels.h"

namespace tadm {
namespace {

// Lexicographic "better" for (value desc, index asc).
__device__ __forceinline__ bool better(float va, int ia, float vb, int ib) {
  return va > vb || (va == vb && ia >= 0 && (ib < 0 || ia < ib));
}

template <int NT>
__device__ __forceinline__ void block_argmax(float& v, int& i, float* sv, int* si) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float v2 = __shfl_xor_sync(0xffffffffu, v, o);
    const int i2 = __shfl_xor_sync(0xffffffffu, i, o);
    if (better(v2, i2, v, i)) { v = v2; i = i2; }
  }
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();
  if (lane == 0) { sv[w] = v; si[w] = i; }
  __syncthreads();
  if (w == 0) {
    v = lane < NT / 32 ? sv[lane] : -INFINITY;
    i = lane < NT / 32 ? si[lane] : -1;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float v2 = __shfl_xor_sync(0xffffffffu, v, o);
      const int i2 = __shfl_xor_sync(0xffffffffu, i, o);
      if (better(v2, i2, v, i)) { v = v2; i = i2; }
    }
    if (lane == 0) { sv[0] = v; si[0] = i; }
  }
  __syncthreads();
  v = sv[0];
  i = si[0];
}

// One block per row of materialised fp32 logits.
__global__ void __launch_bounds__(256) confidence_kernel(const float* __restrict__ logits, int vocab, int ld,
                                                         int mask_id, float* __restrict__ conf,
                                                         int32_t* __restrict__ tok) {
  pdl_enter();
  __shared__ float sv[32];
  __shared__ int si[32];
  const float* l = logits + static_cast<size_t>(blockIdx.x) * ld;
  float best = -INFINITY;
  int arg = -1;
  for (int j = threadIdx.x; j < vocab; j += 256) {
    const float x = l[j];
    if (j != mask_id && better(x, j, best, arg)) { best = x; arg = j; }
  }
  block_argmax<256>(best, arg, sv, si);
  float s = 0.0f;
  for (int j = threadIdx.x; j < vocab; j += 256)
    if (j != mask_id) s += expf(l[j] - best);
  s = warp_sum(s);
  __syncthreads();
  if ((threadIdx.x & 31) == 0) sv[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.0f;
    for (int w = 0; w < 8; ++w) t += sv[w];
    conf[blockIdx.x] = 1.0f / t;
    tok[blockIdx.x] = arg;
  }
}

// One warp per row: merge the per-column-tile (max, sum exp, argmax) partials
// written by the output-head GEMM epilogue.
__global__ void combine_kernel(const float* __restrict__ part, int rows, int n_tiles, float* __restrict__ conf,
                               int32_t* __restrict__ tok, const int32_t* __restrict__ rows_idx) {
  pdl_enter();
  const int r = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (r >= rows) return;
  const float* p = part + static_cast<size_t>(r) * n_tiles * 3;
  float mx = -INFINITY;
  int arg = -1;
  for (int t = lane; t < n_tiles; t += 32) {
    const float m = p[3 * t];
    const int i = __float_as_int(p[3 * t + 2]);
    if (i >= 0 && better(m, i, mx, arg)) { mx = m; arg = i; }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, mx, o);
    const int i2 = __shfl_xor_sync(0xffffffffu, arg, o);
    if (better(m2, i2, mx, arg)) { mx = m2; arg = i2; }
  }
  float s = 0.0f;
  for (int t = lane; t < n_tiles; t += 32) {
    const float m = p[3 * t];
    if (__float_as_int(p[3 * t + 2]) >= 0) s += p[3 * t + 1] * expf(m - mx);
  }
  s = warp_sum(s);
  if (lane == 0) {
    const int dst = rows_idx ? rows_idx[r] : r;   // compacted rows scatter back to their positions
    conf[dst] = 1.0f / s;
    tok[dst] = arg;
  }
}

// One block per sequence: ordered list of the rows that still hold MASK.
__global__ void __launch_bounds__(256) masked_rows_kernel(const int32_t* __restrict__ z, int ldz, int rows,
                                                          int mask_id, int per_seq, int32_t* __restrict__ idx,
                                                          float* __restrict__ conf) {
  pdl_enter();
  __shared__ int base;
  __shared__ int wsum[8];
  const int b = blockIdx.x;
  const int32_t* zb = z + static_cast<size_t>(b) * ldz;
  if (threadIdx.x == 0) base = 0;
  __syncthreads();
  for (int r0 = 0; r0 < rows; r0 += 256) {
    const int r = r0 + threadIdx.x;
    const bool m = r < rows && zb[r] == mask_id;
    if (r < rows) conf[static_cast<size_t>(b) * rows + r] = -INFINITY;
    const unsigned ballot = __ballot_sync(0xffffffffu, m);
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    if (lane == 0) wsum[w] = __popc(ballot);
    __syncthreads();
    int before = base;
    for (int i = 0; i < w; ++i) before += wsum[i];
    const int j = before + __popc(ballot & ((1u << lane) - 1u));
    if (m && j < per_seq) idx[static_cast<size_t>(b) * per_seq + j] = b * rows + r;
    __syncthreads();
    if (threadIdx.x == 0) {
      int t = 0;
      for (int i = 0; i < 8; ++i) t += wsum[i];
      base += t;
    }
    __syncthreads();
  }
  // sequences with fewer masked rows than per_seq: pad with their last row (results overwritten identically)
  if (threadIdx.x == 0)
    for (int j = base; j < per_seq; ++j) idx[static_cast<size_t>(b) * per_seq + j] = b * rows + (rows - 1);
}

// One block per sequence: k rounds of a block-wide (conf desc, pos asc) argmax
// over the positions that still hold MASK; each winner takes its token, which
// also removes it from the candidates of the next round.
__global__ void __launch_bounds__(256) topk_kernel(int32_t* __restrict__ z, int ldz, const float* __restrict__ conf,
                                                   const int32_t* __restrict__ tok, int rows, int k, int mask_id,
                                                   int32_t* __restrict__ selected) {
  pdl_enter();
  __shared__ float sv[32];
  __shared__ int si[32];
  const int b = blockIdx.x;
  int32_t* zb = z + static_cast<size_t>(b) * ldz;
  const float* cb = conf + static_cast<size_t>(b) * rows;
  const int32_t* tb = tok + static_cast<size_t>(b) * rows;
  int32_t* sel = selected ? selected + static_cast<size_t>(b) * k : nullptr;
  for (int j = 0; j < k; ++j) {
    float v = -INFINITY;
    int idx = -1;
    for (int r = threadIdx.x; r < rows; r += 256)
      if (zb[r] == mask_id && better(cb[r], r, v, idx)) { v = cb[r]; idx = r; }
    block_argmax<256>(v, idx, sv, si);
    if (threadIdx.x == 0) {
      if (idx >= 0) zb[idx] = tb[idx];
      if (sel) sel[j] = idx;   // -1 once no candidate is left
    }
    __syncthreads();
    if (idx < 0) {
      if (sel)
        for (int jj = j + 1 + threadIdx.x; jj < k; jj += 256) sel[jj] = -1;
      break;
    }
  }
}

inline const char* err() {
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? nullptr : cudaGetErrorString(e);
}
}  // namespace

const char* confidence_rows(const float* logits, int rows, int vocab, int ld, int mask_id, float* conf, int32_t* tok,
                            cudaStream_t s) {
  if (rows <= 0) return nullptr;
  launch_pdl(confidence_kernel, rows, 256, 0, s, logits, vocab, ld, mask_id, conf, tok);
  return err();
}

const char* combine_partials(const float* part, int rows, int n_tiles, float* conf, int32_t* tok, cudaStream_t s,
                             const int32_t* rows_idx) {
  if (rows <= 0) return nullptr;
  launch_pdl(combine_kernel, (rows + 7) / 8, 256, 0, s, part, rows, n_tiles, conf, tok, rows_idx);
  return err();
}

const char* masked_rows(const int32_t* z, int ldz, int batch, int rows, int mask_id, int per_seq, int32_t* idx,
                        float* conf, cudaStream_t s) {
  if (batch <= 0 || rows <= 0) return nullptr;
  launch_pdl(masked_rows_kernel, batch, 256, 0, s, z, ldz, rows, mask_id, per_seq, idx, conf);
  return err();
}

const char* topk_unmask(int32_t* z, int ldz, const float* conf, const int32_t* tok, int batch, int rows, int k,
                        int mask_id, int32_t* selected, cudaStream_t s) {
  if (batch <= 0 || rows <= 0 || k <= 0) return nullptr;
  launch_pdl(topk_kernel, batch, 256, 0, s, z, ldz, conf, tok, rows, k, mask_id, selected);
  return err();
}

}  // namespace tadm
