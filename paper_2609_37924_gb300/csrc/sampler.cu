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


// ------------------------------------------------------- entropy-bound sampler
// Alg. 2 (App. C.1).  The draws reuse the Philox stream above: u0 picks the
// categorical draw, u1 the re-noise token floor(u1 (V - 1)) of a rejected
// position; the initial canvas is the re-noise of step T.
__device__ __forceinline__ int eb_noise_token(uint64_t seed, int step, int B, int R, int b, int r, int vocab) {
  float u[3];
  remdm_draws(seed, step, B, R, b, r, u);
  const uint64_t k = static_cast<uint64_t>(u[1] * 16777216.0f);   // exact: u1 = k * 2^-24
  return static_cast<int>((k * static_cast<uint64_t>(vocab - 1)) >> 24);
}

__global__ void eb_noise_kernel(int32_t* __restrict__ z, int ldz, int B, int R, int first, int vocab, uint64_t seed,
                                int step) {
  pdl_enter();
  const int G = R - first;
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= B * G) return;
  const int b = i / G, r = first + (i - b * G);
  z[static_cast<size_t>(b) * ldz + r] = eb_noise_token(seed, step, B, R, b, r, vocab);
}

// idx[b * G + g] = b * R + first + g: the canvas rows of the generated positions
__global__ void eb_rows_kernel(int32_t* __restrict__ idx, int B, int R, int first) {
  pdl_enter();
  const int G = R - first;
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= B * G) return;
  const int b = i / G;
  idx[i] = b * R + first + (i - b * G);
}

// One block per generated position j = b * G + g (canvas row first + g) of
// Alg. 2's step, reading the fp32 logits once:
//  - the row max and argmax (lowest id among equal logits, MASK excluded)
//    come from the output head's per-tile partials when `part` is given
//    (the same fp32 values the head wrote as logits), else from a first
//    pass over the row; last (n = 1): z takes the argmax, nothing else runs;
//  - each warp owns a contiguous segment of the row and sums, with
//    coalesced vector loads, e_v = exp(a_v), a_v = (l_v - max) / tau (0 for
//    MASK), into Z and W = sum e_v a_v; q[j, v] = e_v is written when q is
//    given (p = q / Z); H = log Z - W / Z (clamped at +0);
//  - the draw, the first id whose cumulative e exceeds u0 Z: the segment
//    holding it from the warps' sums in order, then one block-wide re-read
//    of that segment (each thread a contiguous sub-range, a block scan, one
//    thread's walk);
//  - outputs: z (the draw), H[j], Zs[j] = Z (optional).
// VEC = 4: float4 loads (vocab, ld, ldq multiples of 4, 16-byte aligned rows).
template <int NT, int VEC>
__global__ void __launch_bounds__(NT) eb_row_kernel(const float* __restrict__ logits, int ld, int G, int first,
                                                    int32_t* __restrict__ z, int ldz, int B, int R, int vocab,
                                                    int mask_id, float inv_tau, int last, uint64_t seed, int step,
                                                    const float* __restrict__ part, int n_tiles,
                                                    void* __restrict__ q, int q_bf16, int ldq,
                                                    float* __restrict__ H, float* __restrict__ Zs) {
  pdl_enter();
  constexpr int NW = NT / 32, U = 4;
  __shared__ float sv[32], segZ[NW], segW[NW], wsc[NW];
  __shared__ int si[32], sh_seg, sh_pick, sh_last;
  __shared__ float sh_goal;
  const int j = blockIdx.x, tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  const int b = j / G, r = first + (j - b * G);
  const float* L = logits + static_cast<size_t>(j) * ld;
  int32_t* zp = z + static_cast<size_t>(b) * ldz + r;
  float mx = -INFINITY;
  int am = -1;
  if (part) {
    const float* pr = part + static_cast<size_t>(j) * n_tiles * 3;
    for (int t = tid; t < n_tiles; t += NT) {
      const int i = __float_as_int(pr[3 * t + 2]);
      if (i >= 0 && better(pr[3 * t], i, mx, am)) { mx = pr[3 * t]; am = i; }
    }
  } else {
    for (int v0 = tid * VEC; v0 < vocab; v0 += NT * VEC * U) {
      float x[U][VEC];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int v = v0 + u * NT * VEC;
        if (v < vocab) {
          if constexpr (VEC == 4) {
            const float4 t = *reinterpret_cast<const float4*>(L + v);
            x[u][0] = t.x, x[u][1] = t.y, x[u][2] = t.z, x[u][3] = t.w;
          } else {
            x[u][0] = L[v];
          }
        }
      }
#pragma unroll
      for (int u = 0; u < U; ++u)
#pragma unroll
        for (int k = 0; k < VEC; ++k) {
          const int v = v0 + u * NT * VEC + k;
          if (v < vocab && v != mask_id && better(x[u][k], v, mx, am)) { mx = x[u][k]; am = v; }
        }
    }
  }
  block_argmax<NT>(mx, am, sv, si);
  if (last) {
    if (tid == 0) *zp = am;
    return;
  }
  // warp segments: S floats each (a multiple of 4), the last one shorter
  const int S = (vocab + NW * 4 - 1) / (NW * 4) * 4;
  auto e_of = [&](float l, int v) { return v == mask_id ? 0.0f : expf((l - mx) * inv_tau); };
  {
    const int lo = w * S, hi = min(vocab, lo + S);
    float Z = 0.0f, W = 0.0f;
    for (int v0 = lo + lane * VEC; v0 < hi; v0 += 32 * VEC * U) {
      float x[U][VEC];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int v = v0 + u * 32 * VEC;
        if (v < hi) {
          if constexpr (VEC == 4) {
            const float4 t = *reinterpret_cast<const float4*>(L + v);
            x[u][0] = t.x, x[u][1] = t.y, x[u][2] = t.z, x[u][3] = t.w;
          } else {
            x[u][0] = L[v];
          }
        }
      }
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int v = v0 + u * 32 * VEC;
        if (v >= hi) continue;
        float e[VEC];
#pragma unroll
        for (int k = 0; k < VEC; ++k) {
          const float a = (x[u][k] - mx) * inv_tau;
          e[k] = v + k == mask_id ? 0.0f : expf(a);
          if (e[k] > 0.0f) {
            Z += e[k];
            W = fmaf(e[k], a, W);
          }
        }
        if (q) {
          if (q_bf16) {
            bf16* o = static_cast<bf16*>(q) + static_cast<size_t>(j) * ldq + v;
            if constexpr (VEC == 4) {
              __nv_bfloat162 p0 = __floats2bfloat162_rn(e[0], e[1]), p1 = __floats2bfloat162_rn(e[2], e[3]);
              uint2 pk;
              pk.x = *reinterpret_cast<uint32_t*>(&p0);
              pk.y = *reinterpret_cast<uint32_t*>(&p1);
              *reinterpret_cast<uint2*>(o) = pk;
            } else {
              o[0] = __float2bfloat16_rn(e[0]);
            }
          } else {
            float* o = static_cast<float*>(q) + static_cast<size_t>(j) * ldq + v;
            if constexpr (VEC == 4) *reinterpret_cast<float4*>(o) = make_float4(e[0], e[1], e[2], e[3]);
            else o[0] = e[0];
          }
        }
      }
    }
    // fixed-order warp sums (the segment sums of the draw)
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      Z += __shfl_xor_sync(0xffffffffu, Z, o);
      W += __shfl_xor_sync(0xffffffffu, W, o);
    }
    if (lane == 0) {
      segZ[w] = Z;
      segW[w] = W;
    }
  }
  __syncthreads();
  if (tid == 0) {
    float u[3];
    remdm_draws(seed, step, B, R, b, r, u);
    float Zt = 0.0f, Wt = 0.0f;
    for (int i = 0; i < NW; ++i) {
      Zt += segZ[i];
      Wt += segW[i];
    }
    const float goal = u[0] * Zt;
    float c = 0.0f;
    int seg = -1, lastseg = -1;
    float before = 0.0f;
    for (int i = 0; i < NW; ++i) {
      if (segZ[i] > 0.0f) {
        if (seg < 0 && c + segZ[i] > goal) {
          seg = i;
          before = c;
        }
        lastseg = i;
      }
      c += segZ[i];
    }
    if (seg < 0) {                                  // rounding left the goal past every segment: the last one
      seg = lastseg;
      before = c - segZ[lastseg >= 0 ? lastseg : 0];
    }
    sh_seg = seg;
    sh_goal = goal - before;
    sh_pick = -1;
    sh_last = -1;
    const float ent = logf(Zt) - Wt / Zt;
    H[j] = ent > 0.0f ? ent : 0.0f;                 // rounding below 0 (and -0) -> +0: keys sort by bits
    if (Zs) Zs[j] = Zt;
  }
  __syncthreads();
  const int seg = sh_seg;
  if (seg >= 0) {
    const int lo = seg * S, hi = min(vocab, lo + S);
    const int c = (hi - lo + NT - 1) / NT, a0 = min(hi, lo + tid * c), a1 = min(hi, a0 + c);
    float mine = 0.0f;
    int lastv = -1;
    for (int v = a0; v < a1; ++v) {
      const float e = e_of(L[v], v);
      mine += e;
      if (e > 0.0f) lastv = v;
    }
    // block inclusive scan of the sub-range sums (warp shuffles, then the warp
    // totals); each thread's interval starts exactly where its predecessor's ends
    float inc = mine;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float t = __shfl_up_sync(0xffffffffu, inc, o);
      if (lane >= o) inc += t;
    }
    float exc = __shfl_up_sync(0xffffffffu, inc, 1);
    if (lane == 0) exc = 0.0f;
    if (lane == 31) wsc[w] = inc;
    if (lastv >= 0) atomicMax(&sh_last, lastv);
    __syncthreads();
    float wb = 0.0f;
    for (int i = 0; i < w; ++i) wb += wsc[i];
    inc += wb;
    const float before = exc + wb, goal = sh_goal;
    if (mine > 0.0f && before <= goal && goal < inc) {
      float run = before;
      int got = -1;
      for (int v = a0; v < a1; ++v) {
        const float e = e_of(L[v], v);
        if (e > 0.0f) {
          run += e;
          if (run > goal) {
            got = v;
            break;
          }
        }
      }
      sh_pick = got >= 0 ? got : lastv;             // rounding kept the walk at or below the goal: the range's last
    }
    __syncthreads();
  }
  if (tid == 0) {
    int v = seg >= 0 ? sh_pick : -1;
    if (v < 0 && seg >= 0) v = sh_last;             // no sub-range held the goal: the segment's last token
    *zp = v < 0 ? am : v;
  }
}

// One block per sequence: the G entropies sorted ascending (ties to the lower
// position) as 64-bit keys (H bits, position) by a bitonic sort in shared
// memory (H >= 0, so the fp32 bit patterns order like the values); C_m of
// the sorted order by an fp64 block scan; position pi_m keeps its draw when
// C_m - H_{pi_m} <= eta (H_{pi_m} = M_m in ascending order), otherwise it
// takes the re-noise token.  keys: n2 = next power of two >= G entries.
template <int NT>
__global__ void __launch_bounds__(NT) eb_accept_kernel(const float* __restrict__ H, int G, int n2, int first,
                                                       int32_t* __restrict__ z, int ldz, int B, int R, int vocab,
                                                       double eta, uint64_t seed, int step) {
  pdl_enter();
  extern __shared__ unsigned long long keys[];
  __shared__ double part[NT];
  const int b = blockIdx.x, tid = threadIdx.x;
  for (int i = tid; i < n2; i += NT)
    keys[i] = i < G ? (static_cast<unsigned long long>(__float_as_uint(H[static_cast<size_t>(b) * G + i])) << 32) |
                          static_cast<unsigned>(i)
                    : ~0ull;
  __syncthreads();
  for (int k = 2; k <= n2; k <<= 1)
    for (int jj = k >> 1; jj > 0; jj >>= 1) {
      for (int i = tid; i < n2; i += NT) {
        const int l = i ^ jj;
        if (l > i) {
          const unsigned long long a = keys[i], c = keys[l];
          const bool up = (i & k) == 0;
          if ((a > c) == up) {
            keys[i] = c;
            keys[l] = a;
          }
        }
      }
      __syncthreads();
    }
  const int per = (n2 + NT - 1) / NT, m0 = tid * per, m1 = min(n2, m0 + per);
  double mine = 0.0;
  for (int m = m0; m < m1; ++m)
    if (static_cast<unsigned>(keys[m]) < static_cast<unsigned>(G)) mine += __uint_as_float(keys[m] >> 32);
  part[tid] = mine;
  __syncthreads();
  for (int o = 1; o < NT; o <<= 1) {               // inclusive scan of the range sums
    const double add = tid >= o ? part[tid - o] : 0.0;
    __syncthreads();
    part[tid] += add;
    __syncthreads();
  }
  double c = tid > 0 ? part[tid - 1] : 0.0;
  for (int m = m0; m < m1; ++m) {
    const unsigned g = static_cast<unsigned>(keys[m]);
    if (g >= static_cast<unsigned>(G)) continue;
    const double h = __uint_as_float(keys[m] >> 32);
    c += h;
    if (!(c - h <= eta)) {
      const int r = first + static_cast<int>(g);
      z[static_cast<size_t>(b) * ldz + r] = eb_noise_token(seed, step, B, R, b, r, vocab);
    }
  }
}

// E^T: out[c, r] = in[r, c] for a rows x cols matrix (32 x 32 shared tiles;
// T is the element's bit container: float or uint16_t for bf16)
template <class T>
__global__ void transpose_kernel(const T* __restrict__ in, int rows, int cols, T* __restrict__ out) {
  pdl_enter();
  __shared__ T t[32][33];
  const int r0 = blockIdx.x * 32, c0 = blockIdx.y * 32;
  for (int y = threadIdx.y; y < 32; y += 8) {
    const int r = r0 + y, c = c0 + threadIdx.x;
    if (r < rows && c < cols) t[y][threadIdx.x] = in[static_cast<size_t>(r) * cols + c];
  }
  __syncthreads();
  for (int y = threadIdx.y; y < 32; y += 8) {
    const int c = c0 + y, r = r0 + threadIdx.x;
    if (r < rows && c < cols) out[static_cast<size_t>(c) * rows + r] = t[threadIdx.x][y];
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

const char* eb_noise(int32_t* z, int ldz, int B, int R, int first, int vocab, uint64_t seed, int step, cudaStream_t s) {
  const int n = B * (R - first);
  if (n <= 0) return nullptr;
  launch_pdl(eb_noise_kernel, (n + 255) / 256, 256, 0, s, z, ldz, B, R, first, vocab, seed, step);
  return err();
}

const char* eb_rows(int32_t* idx, int B, int R, int first, cudaStream_t s) {
  const int n = B * (R - first);
  if (n <= 0) return nullptr;
  launch_pdl(eb_rows_kernel, (n + 255) / 256, 256, 0, s, idx, B, R, first);
  return err();
}

const char* eb_row(const float* logits, int ld, int B, int R, int first, int32_t* z, int ldz, int vocab, int mask_id,
                   float inv_tau, int last, uint64_t seed, int step, const float* part, int n_tiles, void* q,
                   int q_bf16, int ldq, float* H, float* Zs, cudaStream_t s) {
  const int G = R - first, n = B * G;
  if (n <= 0) return nullptr;
  const bool vec = vocab % 4 == 0 && ld % 4 == 0 && reinterpret_cast<uintptr_t>(logits) % 16 == 0 &&
                   (!q || (ldq % 4 == 0 && reinterpret_cast<uintptr_t>(q) % 16 == 0));
  if (vec)
    launch_pdl(eb_row_kernel<512, 4>, n, 512, 0, s, logits, ld, G, first, z, ldz, B, R, vocab, mask_id, inv_tau, last,
               seed, step, part, n_tiles, q, q_bf16, ldq, H, Zs);
  else
    launch_pdl(eb_row_kernel<512, 1>, n, 512, 0, s, logits, ld, G, first, z, ldz, B, R, vocab, mask_id, inv_tau, last,
               seed, step, part, n_tiles, q, q_bf16, ldq, H, Zs);
  return err();
}

int eb_max_gen() { return 16384; }

const char* eb_accept(const float* H, int B, int R, int first, int32_t* z, int ldz, int vocab, double eta,
                      uint64_t seed, int step, cudaStream_t s) {
  const int G = R - first;
  if (B <= 0 || G <= 0) return nullptr;
  if (G > eb_max_gen()) return "entropy-bound sampler: more than 16384 generated positions per sequence";
  int n2 = 1;
  while (n2 < G) n2 <<= 1;
  static bool attr = false;
  if (!attr) {
    if (cudaFuncSetAttribute(eb_accept_kernel<1024>, cudaFuncAttributeMaxDynamicSharedMemorySize, 16384 * 8) !=
        cudaSuccess)
      return "entropy-bound accept smem attribute failed";
    attr = true;
  }
  launch_pdl(eb_accept_kernel<1024>, B, 1024, static_cast<size_t>(n2) * 8, s, H, G, n2, first, z, ldz, B, R, vocab,
             eta, seed, step);
  return err();
}

const char* transpose(const void* in, int rows, int cols, int bf16, void* out, cudaStream_t s) {
  if (rows <= 0 || cols <= 0) return nullptr;
  if ((cols + 31) / 32 > 65535) return "transpose: too many columns";
  const dim3 grid((rows + 31) / 32, (cols + 31) / 32), block(32, 8);
  if (bf16)
    launch_pdl(transpose_kernel<uint16_t>, grid, block, 0, s, static_cast<const uint16_t*>(in), rows, cols,
               static_cast<uint16_t*>(out));
  else
    launch_pdl(transpose_kernel<float>, grid, block, 0, s, static_cast<const float*>(in), rows, cols,
               static_cast<float*>(out));
  return err();
}

}  // namespace tadm
