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
// ------------------------------------------------------------ ReMDM sampler
// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11): ten rounds of two
// 32x32 -> 64-bit multiplies with the published multipliers and Weyl key
// increments.
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint2 k) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint32_t lo0 = 0xD2511F53u * c.x, hi0 = __umulhi(0xD2511F53u, c.x);
    const uint32_t lo1 = 0xCD9E8D57u * c.z, hi1 = __umulhi(0xCD9E8D57u, c.z);
    c = make_uint4(hi1 ^ c.y ^ k.x, lo1, hi0 ^ c.w ^ k.y, lo0);
    k.x += 0x9E3779B9u;
    k.y += 0xBB67AE85u;
  }
  return c;
}

constexpr uint32_t kRemdmStream = 0x52454D44u;   // "REMD"

// The three draws of canvas position (b, r) at reverse step n: Philox block
// (n * B + b) * R + r of the REMD stream, uniform j = (word j >> 8) * 2^-24.
__device__ __forceinline__ void remdm_draws(uint64_t seed, int step, int B, int R, int b, int r, float (&u)[3]) {
  const uint64_t blk = (static_cast<uint64_t>(step) * B + b) * static_cast<uint64_t>(R) + r;
  const uint4 w = philox4x32_10(make_uint4(static_cast<uint32_t>(blk), static_cast<uint32_t>(blk >> 32), kRemdmStream, 0u),
                                make_uint2(static_cast<uint32_t>(seed), static_cast<uint32_t>(seed >> 32)));
  u[0] = static_cast<float>(w.x >> 8) * (1.0f / 16777216.0f);
  u[1] = static_cast<float>(w.y >> 8) * (1.0f / 16777216.0f);
  u[2] = static_cast<float>(w.z >> 8) * (1.0f / 16777216.0f);
}

__global__ void remdm_uniforms_kernel(uint64_t seed, int step, int B, int R, float* __restrict__ out) {
  pdl_enter();
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= B * R) return;
  float u[3];
  remdm_draws(seed, step, B, R, i / R, i % R, u);
  out[3 * i] = u[0];
  out[3 * i + 1] = u[1];
  out[3 * i + 2] = u[2];
}

// One thread per canvas position of the active rows: action 0 keep, 1 remask
// (a generated token, u0 < sigma: written as MASK here), 2 unmask (a masked
// position, u1 < p_unmask: its token is drawn by remdm_sample_kernel).  The
// comparisons are in fp64, exactly as the oracle takes them.
__global__ void remdm_decide_kernel(int32_t* __restrict__ z, int ldz, int B, int R, int first_gen, int mask_id,
                                    double sigma, double p_unmask, uint64_t seed, int step, int32_t* __restrict__ act) {
  pdl_enter();
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= B * R) return;
  const int b = i / R, r = i - (i / R) * R;
  int a = 0;
  if (r >= first_gen) {
    float u[3];
    remdm_draws(seed, step, B, R, b, r, u);
    int32_t* zp = z + static_cast<size_t>(b) * ldz + r;
    if (*zp != mask_id) {
      if (static_cast<double>(u[0]) < sigma) {
        a = 1;
        *zp = mask_id;
      }
    } else if (static_cast<double>(u[1]) < p_unmask) {
      a = 2;
    }
  }
  act[i] = a;
}

// One 1024-thread block: the rows with action 2 in row order, idx[0 .. count),
// *count; entries count .. bound-1 repeat the first such row (or row 0), so
// every entry names a valid row for gathers sized by the bound.
__global__ void __launch_bounds__(1024) remdm_rows_kernel(const int32_t* __restrict__ act, int n, int bound,
                                                          int32_t* __restrict__ idx, int* __restrict__ count) {
  pdl_enter();
  __shared__ int wsum[32];
  __shared__ int base;
  if (threadIdx.x == 0) base = 0;
  __syncthreads();
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  for (int r0 = 0; r0 < n; r0 += 1024) {
    const int r = r0 + threadIdx.x;
    const bool on = r < n && act[r] == 2;
    const unsigned ballot = __ballot_sync(0xffffffffu, on);
    if (lane == 0) wsum[w] = __popc(ballot);
    __syncthreads();
    int before = base;
    for (int i = 0; i < w; ++i) before += wsum[i];
    const int j = before + __popc(ballot & ((1u << lane) - 1u));
    if (on && j < bound) idx[j] = r;
    __syncthreads();
    if (threadIdx.x == 0) {
      int t = 0;
      for (int i = 0; i < 32; ++i) t += wsum[i];
      base += t;
    }
    __syncthreads();
  }
  const int cnt = min(base, bound);
  __syncthreads();
  const int fill = cnt > 0 ? idx[0] : 0;
  for (int j = cnt + threadIdx.x; j < bound; j += 1024) idx[j] = fill;
  if (threadIdx.x == 0) *count = cnt;
}

template <int NT>
__device__ __forceinline__ float block_sum_f(float v, float* red) {
  v = warp_sum(v);
  __syncthreads();
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
  __syncthreads();
  float t = 0.0f;
#pragma unroll
  for (int w = 0; w < NT / 32; ++w) t += red[w];
  return t;
}

// One block per logits row j (canvas row idx[j], or j): for rows whose action
// is 2, the nucleus (top-p) token of softmax over ids != MASK, by inverse CDF
// in id order within the nucleus.  The nucleus threshold is the largest fp32
// tau with sum_{q_v >= tau} q_v >= top_p * sum q (q = exp(l - max)), found by
// bisection on the bit patterns of tau in [0, 1]; each thread owns a
// contiguous id range, so the id-order prefix sum is a block scan of range
// sums followed by one thread's walk of its range.
template <int NT>
__global__ void __launch_bounds__(NT) remdm_sample_kernel(const float* __restrict__ logits, int ld, int n_rows,
                                                          const int32_t* __restrict__ idx, const int32_t* __restrict__ act,
                                                          int32_t* __restrict__ z, int ldz, int B, int R, int vocab,
                                                          int mask_id, float top_p, uint64_t seed, int step,
                                                          const int* __restrict__ count) {
  pdl_enter();
  __shared__ float red[NT / 32];
  __shared__ float scan[NT];
  __shared__ int pick;
  const int j = blockIdx.x;
  if (j >= n_rows || (count && j >= *count)) return;
  const int row = idx ? idx[j] : j;
  if (act[row] != 2) return;                     // uniform across the block
  const int b = row / R, r = row - (row / R) * R;
  const float* L = logits + static_cast<size_t>(j) * ld;
  const int tid = threadIdx.x;
  const int chunk = (vocab + NT - 1) / NT, v0 = tid * chunk, v1 = min(vocab, v0 + chunk);
  float mx = -INFINITY;
  for (int v = v0; v < v1; ++v)
    if (v != mask_id) mx = fmaxf(mx, L[v]);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  __syncthreads();
  if ((tid & 31) == 0) red[tid >> 5] = mx;
  __syncthreads();
  mx = red[0];
#pragma unroll
  for (int w = 1; w < NT / 32; ++w) mx = fmaxf(mx, red[w]);
  // mass at or above tau (tau = 0: the whole mass)
  auto mass_from = [&](float tau) {
    float acc = 0.0f;
    for (int v = v0; v < v1; ++v) {
      const float q = v == mask_id ? 0.0f : expf(L[v] - mx);
      acc += q >= tau && q > 0.0f ? q : 0.0f;
    }
    return block_sum_f<NT>(acc, red);
  };
  const float total = mass_from(0.0f);
  const float target = top_p * total;
  uint32_t lo = 0u, hi = 0x3F800001u;            // mass_from(lo) >= target > mass_from(hi)
  while (hi - lo > 1u) {
    const uint32_t mid = lo + (hi - lo) / 2u;
    if (mass_from(__uint_as_float(mid)) >= target) lo = mid;
    else hi = mid;
  }
  const float tau = __uint_as_float(lo);
  // id-order inverse CDF within the nucleus
  float mine = 0.0f;
  for (int v = v0; v < v1; ++v) {
    const float q = v == mask_id ? 0.0f : expf(L[v] - mx);
    mine += q >= tau && q > 0.0f ? q : 0.0f;
  }
  scan[tid] = mine;
  if (tid == 0) pick = -1;
  __syncthreads();
  for (int o = 1; o < NT; o <<= 1) {             // inclusive scan of the range sums (fixed order)
    const float add = tid >= o ? scan[tid - o] : 0.0f;
    __syncthreads();
    scan[tid] += add;
    __syncthreads();
  }
  float u[3];
  remdm_draws(seed, step, B, R, b, r, u);
  const float zn = scan[NT - 1];
  const float goal = u[2] * zn;
  const float before = tid > 0 ? scan[tid - 1] : 0.0f;
  if (mine > 0.0f && before <= goal && goal < scan[tid]) {
    // the walk re-adds this range in the same order; if rounding keeps it
    // at or below the goal, the range's last nucleus token is the draw
    float c = before;
    int last = -1, got = -1;
    for (int v = v0; v < v1; ++v) {
      const float q = v == mask_id ? 0.0f : expf(L[v] - mx);
      if (q >= tau && q > 0.0f) {
        last = v;
        c += q;
        if (c > goal) {
          got = v;
          break;
        }
      }
    }
    pick = got >= 0 ? got : last;
  }
  __syncthreads();
  if (tid == 0) {
    int v = pick;
    if (v < 0) {                                  // rounding left the goal past the last range: its last token
      for (int t = NT - 1; t >= 0 && v < 0; --t)
        if ((t > 0 ? scan[t] - scan[t - 1] : scan[0]) > 0.0f) {
          const int a0 = t * chunk, a1 = min(vocab, a0 + chunk);
          for (int w = a1 - 1; w >= a0; --w)
            if (w != mask_id && expf(L[w] - mx) >= tau && expf(L[w] - mx) > 0.0f) { v = w; break; }
        }
    }
    z[static_cast<size_t>(b) * ldz + r] = v;
  }
}

// remdm_sample_kernel with the row's probabilities staged once in shared
// memory (q_v = exp(l_v - max), 0 for MASK; vocab * 4 bytes of dynamic
// shared memory): the bisection sums read shared memory with a strided
// (bank-conflict-free) assignment, the id-order draw uses contiguous ranges.
template <int NT>
__global__ void __launch_bounds__(NT) remdm_sample_smem_kernel(const float* __restrict__ logits, int ld, int n_rows,
                                                               const int32_t* __restrict__ idx,
                                                               const int32_t* __restrict__ act, int32_t* __restrict__ z,
                                                               int ldz, int B, int R, int vocab, int mask_id,
                                                               float top_p, uint64_t seed, int step,
                                                               const int* __restrict__ count) {
  pdl_enter();
  extern __shared__ float qs[];
  __shared__ float red[NT / 32];
  __shared__ float scan[NT];
  __shared__ int pick;
  const int j = blockIdx.x;
  if (j >= n_rows || (count && j >= *count)) return;
  const int row = idx ? idx[j] : j;
  if (act[row] != 2) return;
  const int b = row / R, r = row - (row / R) * R;
  const float* L = logits + static_cast<size_t>(j) * ld;
  const int tid = threadIdx.x;
  float mx = -INFINITY;
  for (int v = tid; v < vocab; v += NT) {
    const float l = L[v];
    qs[v] = l;
    if (v != mask_id) mx = fmaxf(mx, l);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  if ((tid & 31) == 0) red[tid >> 5] = mx;
  __syncthreads();
  mx = red[0];
#pragma unroll
  for (int w = 1; w < NT / 32; ++w) mx = fmaxf(mx, red[w]);
  for (int v = tid; v < vocab; v += NT) qs[v] = v == mask_id ? 0.0f : expf(qs[v] - mx);
  auto mass_from = [&](float tau) {
    float acc = 0.0f;
    for (int v = tid; v < vocab; v += NT) {
      const float q = qs[v];
      acc += q >= tau && q > 0.0f ? q : 0.0f;
    }
    return block_sum_f<NT>(acc, red);
  };
  const float total = mass_from(0.0f);
  const float target = top_p * total;
  uint32_t lo = 0u, hi = 0x3F800001u;
  while (hi - lo > 1u) {
    const uint32_t mid = lo + (hi - lo) / 2u;
    if (mass_from(__uint_as_float(mid)) >= target) lo = mid;
    else hi = mid;
  }
  const float tau = __uint_as_float(lo);
  const int chunk = (vocab + NT - 1) / NT, v0 = tid * chunk, v1 = min(vocab, v0 + chunk);
  float mine = 0.0f;
  for (int v = v0; v < v1; ++v) {
    const float q = qs[v];
    mine += q >= tau && q > 0.0f ? q : 0.0f;
  }
  scan[tid] = mine;
  if (tid == 0) pick = -1;
  __syncthreads();
  for (int o = 1; o < NT; o <<= 1) {
    const float add = tid >= o ? scan[tid - o] : 0.0f;
    __syncthreads();
    scan[tid] += add;
    __syncthreads();
  }
  float u[3];
  remdm_draws(seed, step, B, R, b, r, u);
  const float goal = u[2] * scan[NT - 1];
  const float before = tid > 0 ? scan[tid - 1] : 0.0f;
  if (mine > 0.0f && before <= goal && goal < scan[tid]) {
    float c = before;
    int last = -1, got = -1;
    for (int v = v0; v < v1; ++v) {
      const float q = qs[v];
      if (q >= tau && q > 0.0f) {
        last = v;
        c += q;
        if (c > goal) {
          got = v;
          break;
        }
      }
    }
    pick = got >= 0 ? got : last;
  }
  __syncthreads();
  if (tid == 0) {
    int v = pick;
    for (int t = NT - 1; t >= 0 && v < 0; --t)   // rounding left the goal past every range: the last token
      if ((t > 0 ? scan[t] - scan[t - 1] : scan[0]) > 0.0f)
        for (int w = min(vocab, (t + 1) * chunk) - 1; w >= t * chunk; --w)
          if (qs[w] >= tau && qs[w] > 0.0f) { v = w; break; }
    z[static_cast<size_t>(b) * ldz + r] = v;
  }
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

const char* remdm_uniforms(uint64_t seed, int step, int B, int R, float* out, cudaStream_t s) {
  if (B * R <= 0) return nullptr;
  launch_pdl(remdm_uniforms_kernel, (B * R + 255) / 256, 256, 0, s, seed, step, B, R, out);
  return err();
}

const char* remdm_decide(int32_t* z, int ldz, int B, int R, int first_gen, int mask_id, double sigma,
                         double p_unmask, uint64_t seed, int step, int32_t* act, cudaStream_t s) {
  if (B * R <= 0) return nullptr;
  launch_pdl(remdm_decide_kernel, (B * R + 255) / 256, 256, 0, s, z, ldz, B, R, first_gen, mask_id, sigma, p_unmask,
             seed, step, act);
  return err();
}

const char* remdm_sample(const float* logits, int ld, int n_rows, const int32_t* idx, const int32_t* act, int32_t* z,
                         int ldz, int B, int R, int vocab, int mask_id, float top_p, uint64_t seed, int step,
                         cudaStream_t s, const int* count) {
  if (n_rows <= 0) return nullptr;
  const size_t smem = static_cast<size_t>(vocab) * sizeof(float);
  if (smem <= 200u * 1024u) {   // the row's probabilities fit in shared memory
    static bool attr = false;
    if (!attr) {
      if (cudaFuncSetAttribute(remdm_sample_smem_kernel<1024>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               200 * 1024) != cudaSuccess)
        return "sampler smem attribute failed";
      attr = true;
    }
    launch_pdl(remdm_sample_smem_kernel<1024>, n_rows, 1024, smem, s, logits, ld, n_rows, idx, act, z, ldz, B, R,
               vocab, mask_id, top_p, seed, step, count);
  } else {
    launch_pdl(remdm_sample_kernel<256>, n_rows, 256, 0, s, logits, ld, n_rows, idx, act, z, ldz, B, R, vocab,
               mask_id, top_p, seed, step, count);
  }
  return err();
}

const char* remdm_rows(const int32_t* act, int n, int bound, int32_t* idx, int* count, cudaStream_t s) {
  launch_pdl(remdm_rows_kernel, 1, 1024, 0, s, act, n, bound, idx, count);
  return err();
}

}  // namespace tadm
