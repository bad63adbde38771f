// Row-wise kernels of the path (HBM-bound, one warp per row, float4 I/O):
// token-embedding gather (S), RMSNorm ahead of each projection, the two
// LayerNorms that build the fusion input u = [LN(c); LN(h)] and the output
// LayerNorm of the gated-MLP fusion (App. C.2), the RMS scales and feature
// concatenations of the paired-attention fusion (App. C.1), the RoPE table,
// and canvas set-up.
#include <cstdlib>
#include <initializer_list>

#include "kernels.h"

namespace tadm {

bool pdl_enabled() {
  static const bool on = [] {
    const char* e = getenv("TADM_PDL");
    return !(e && e[0] == '0');
  }();
  return on;
}

namespace {

constexpr int WPB = 8;  // warps (rows) per block

template <class T>
__device__ __forceinline__ void store_act(void* out, size_t i, float v);
template <>
__device__ __forceinline__ void store_act<float>(void* out, size_t i, float v) { static_cast<float*>(out)[i] = v; }
template <>
__device__ __forceinline__ void store_act<bf16>(void* out, size_t i, float v) {
  static_cast<bf16*>(out)[i] = __float2bfloat16_rn(v);
}

// act value v at out[i]; with lo_off > 0 (bf16 only) also the rounding
// remainder bf16(v - hi) at out[i + lo_off]: the split (hi + lo) operand of a
// projection whose input is carried at about 16 bits
template <class T>
__device__ __forceinline__ void store_act2(void* out, size_t i, float v, int lo_off);
template <>
__device__ __forceinline__ void store_act2<float>(void* out, size_t i, float v, int) { static_cast<float*>(out)[i] = v; }
template <>
__device__ __forceinline__ void store_act2<bf16>(void* out, size_t i, float v, int lo_off) {
  const bf16 hi = __float2bfloat16_rn(v);
  static_cast<bf16*>(out)[i] = hi;
  if (lo_off > 0) static_cast<bf16*>(out)[i + lo_off] = __float2bfloat16_rn(v - __bfloat162float(hi));
}

__device__ __forceinline__ float ldw(const void* w, int bf, int i) {
  return bf ? __bfloat162float(static_cast<const bf16*>(w)[i]) : static_cast<const float*>(w)[i];
}

__global__ void embed_kernel(const int32_t* __restrict__ z, int ldz, int rows, int M, const void* __restrict__ E,
                             int e_bf16, int d, int vocab, float* __restrict__ out, float* __restrict__ out2,
                             const float* __restrict__ add, int add_first, const float* __restrict__ add_div) {
  pdl_enter();
  const int m = blockIdx.x * WPB + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (m >= M) return;
  const int b = m / rows, r = m - b * rows;
  int tok = z[static_cast<size_t>(b) * ldz + r];
  tok = tok < 0 ? 0 : (tok >= vocab ? vocab - 1 : tok);  // ids are validated by the caller; never read outside E
  float* o = out + static_cast<size_t>(m) * d;
  float* o2 = out2 ? out2 + static_cast<size_t>(m) * d : nullptr;
  const size_t ar = static_cast<size_t>(b) * (rows - add_first) + (r - add_first);
  const float* a = add && r >= add_first ? add + ar * d : nullptr;
  const float sc = a && add_div ? 1.0f / add_div[ar] : 1.0f;
  if (e_bf16) {
    const bf16* e = static_cast<const bf16*>(E) + static_cast<size_t>(tok) * d;
    for (int j = lane * 2; j < d; j += 64) {
      float2 v = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(e + j));
      if (a) {
        const float2 t = *reinterpret_cast<const float2*>(a + j);
        v.x = fmaf(t.x, sc, v.x);
        v.y = fmaf(t.y, sc, v.y);
      }
      *reinterpret_cast<float2*>(o + j) = v;
      if (o2) *reinterpret_cast<float2*>(o2 + j) = v;
    }
  } else {
    const float* e = static_cast<const float*>(E) + static_cast<size_t>(tok) * d;
    for (int j = lane * 4; j < d; j += 128) {
      float4 v = *reinterpret_cast<const float4*>(e + j);
      if (a) {
        const float4 t = *reinterpret_cast<const float4*>(a + j);
        v.x = fmaf(t.x, sc, v.x);
        v.y = fmaf(t.y, sc, v.y);
        v.z = fmaf(t.z, sc, v.z);
        v.w = fmaf(t.w, sc, v.w);
      }
      *reinterpret_cast<float4*>(o + j) = v;
      if (o2) *reinterpret_cast<float4*>(o2 + j) = v;
    }
  }
}

// out = x / sqrt(mean(x^2) + eps) * gain, one 256-thread block per row (few rows)
template <class T>
__global__ void __launch_bounds__(256) rmsnorm_block_kernel(const float* __restrict__ x, int d,
                                                            const void* __restrict__ gain, int w_bf16, float eps,
                                                            void* __restrict__ out, int ldo,
                                                            const int32_t* __restrict__ rows_idx, int lo_off) {
  pdl_enter();
  __shared__ float red[8];
  const int m = blockIdx.x;
  const float* xr = x + static_cast<size_t>(rows_idx ? rows_idx[m] : m) * d;
  float ss = 0.0f;
  for (int j = threadIdx.x * 4; j < d; j += 1024) {
    const float4 v = *reinterpret_cast<const float4*>(xr + j);
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
  ss = warp_sum(ss);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  float tot = 0.0f;
#pragma unroll
  for (int w = 0; w < 8; ++w) tot += red[w];
  const float inv = rsqrtf(tot / static_cast<float>(d) + eps);
  for (int j = threadIdx.x * 4; j < d; j += 1024) {
    const float4 v = *reinterpret_cast<const float4*>(xr + j);
    const size_t o = static_cast<size_t>(m) * ldo + j;
    store_act2<T>(out, o + 0, v.x * inv * ldw(gain, w_bf16, j + 0), lo_off);
    store_act2<T>(out, o + 1, v.y * inv * ldw(gain, w_bf16, j + 1), lo_off);
    store_act2<T>(out, o + 2, v.z * inv * ldw(gain, w_bf16, j + 2), lo_off);
    store_act2<T>(out, o + 3, v.w * inv * ldw(gain, w_bf16, j + 3), lo_off);
  }
}

// out = x / sqrt(mean(x^2) + eps) * gain
template <class T>
__global__ void rmsnorm_kernel(const float* __restrict__ x, int M, int d, const void* __restrict__ gain, int w_bf16,
                               float eps, void* __restrict__ out, int ldo, const int32_t* __restrict__ rows_idx,
                               int lo_off) {
  pdl_enter();
  const int m = blockIdx.x * WPB + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (m >= M) return;
  const float* xr = x + static_cast<size_t>(rows_idx ? rows_idx[m] : m) * d;
  float ss = 0.0f;
  for (int j = lane * 4; j < d; j += 128) {
    const float4 v = *reinterpret_cast<const float4*>(xr + j);
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
  ss = warp_sum(ss);
  const float inv = rsqrtf(ss / static_cast<float>(d) + eps);
  for (int j = lane * 4; j < d; j += 128) {
    const float4 v = *reinterpret_cast<const float4*>(xr + j);
    const size_t o = static_cast<size_t>(m) * ldo + j;
    store_act2<T>(out, o + 0, v.x * inv * ldw(gain, w_bf16, j + 0), lo_off);
    store_act2<T>(out, o + 1, v.y * inv * ldw(gain, w_bf16, j + 1), lo_off);
    store_act2<T>(out, o + 2, v.z * inv * ldw(gain, w_bf16, j + 2), lo_off);
    store_act2<T>(out, o + 3, v.w * inv * ldw(gain, w_bf16, j + 3), lo_off);
  }
}

// out = x / sqrt(mean(x^2) + eps) * gain for d = 256 * NCH: one warp per row,
// the row held in registers (8 consecutive elements per lane and chunk), one
// 16-byte load of 8 gains and one 16-byte store of 8 bf16 outputs per chunk.
// Needs 16-byte aligned x, out (ldo % 8 == 0) and bf16 gains.
template <int NCH>
__global__ void __launch_bounds__(WPB * 32) rmsnorm_reg_kernel(const float* __restrict__ x, int M,
                                                               const bf16* __restrict__ gain, float eps,
                                                               bf16* __restrict__ out, int ldo,
                                                               const int32_t* __restrict__ rows_idx, int lo_off) {
  pdl_enter();
  constexpr int d = 256 * NCH;
  const int m = blockIdx.x * WPB + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (m >= M) return;
  const float* xr = x + static_cast<size_t>(rows_idx ? rows_idx[m] : m) * d;
  float v[NCH][8];
  float ss = 0.0f;
#pragma unroll
  for (int c = 0; c < NCH; ++c) {
    const int j = (c * 32 + lane) * 8;
    const float4 a = *reinterpret_cast<const float4*>(xr + j);
    const float4 b = *reinterpret_cast<const float4*>(xr + j + 4);
    v[c][0] = a.x; v[c][1] = a.y; v[c][2] = a.z; v[c][3] = a.w;
    v[c][4] = b.x; v[c][5] = b.y; v[c][6] = b.z; v[c][7] = b.w;
#pragma unroll
    for (int i = 0; i < 8; ++i) ss = fmaf(v[c][i], v[c][i], ss);
  }
  ss = warp_sum(ss);
  const float inv = rsqrtf(ss / static_cast<float>(d) + eps);
  bf16* orow = out + static_cast<size_t>(m) * ldo;
#pragma unroll
  for (int c = 0; c < NCH; ++c) {
    const int j = (c * 32 + lane) * 8;
    const uint4 graw = *reinterpret_cast<const uint4*>(gain + j);
    const __nv_bfloat162* g2 = reinterpret_cast<const __nv_bfloat162*>(&graw);
    uint32_t packed[4], packed_lo[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float2 g = __bfloat1622float2(g2[q]);
      const float y0 = v[c][2 * q] * inv * g.x, y1 = v[c][2 * q + 1] * inv * g.y;
      __nv_bfloat162 t = __floats2bfloat162_rn(y0, y1);
      packed[q] = *reinterpret_cast<uint32_t*>(&t);
      const float2 th = __bfloat1622float2(t);
      __nv_bfloat162 tl = __floats2bfloat162_rn(y0 - th.x, y1 - th.y);   // remainder of the split operand
      packed_lo[q] = *reinterpret_cast<uint32_t*>(&tl);
    }
    *reinterpret_cast<uint4*>(orow + j) = make_uint4(packed[0], packed[1], packed[2], packed[3]);
    if (lo_off > 0)
      *reinterpret_cast<uint4*>(orow + lo_off + j) = make_uint4(packed_lo[0], packed_lo[1], packed_lo[2], packed_lo[3]);
  }
}

__device__ __forceinline__ void row_mean_var(const float* xr, int d, int lane, float& mean, float& rstd, float eps) {
  float s = 0.0f;
  for (int j = lane * 4; j < d; j += 128) {
    const float4 v = *reinterpret_cast<const float4*>(xr + j);
    s += v.x + v.y + v.z + v.w;
  }
  mean = warp_sum(s) / static_cast<float>(d);
  float q = 0.0f;
  for (int j = lane * 4; j < d; j += 128) {
    const float4 v = *reinterpret_cast<const float4*>(xr + j);
    const float a = v.x - mean, b = v.y - mean, c = v.z - mean, e = v.w - mean;
    q += a * a + b * b + c * c + e * e;
  }
  rstd = rsqrtf(warp_sum(q) / static_cast<float>(d) + eps);
}

// u[m] = [LN(c[m]) * wc + bc ; LN(h[m]) * wh + bh]   (act, [M, 2d])
template <class T>
__global__ void ln_pair_kernel(const float* __restrict__ c, const float* __restrict__ h, int M, int d,
                               const void* wc, const void* bc, const void* wh, const void* bh, int w_bf16, float eps,
                               void* __restrict__ u) {
  pdl_enter();
  const int m = blockIdx.x * WPB + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (m >= M) return;
  for (int part = 0; part < 2; ++part) {
    const float* xr = (part ? h : c) + static_cast<size_t>(m) * d;
    const void* w = part ? wh : wc;
    const void* b = part ? bh : bc;
    float mean, rstd;
    row_mean_var(xr, d, lane, mean, rstd, eps);
    for (int j = lane; j < d; j += 32)
      store_act<T>(u, static_cast<size_t>(m) * 2 * d + part * d + j,
                   (xr[j] - mean) * rstd * ldw(w, w_bf16, j) + ldw(b, w_bf16, j));
  }
}

// Register-resident LayerNorm of one row of d = 256 NCH columns (one warp per
// row): the lane holds the 8 consecutive values of each 256-column chunk, so
// the row is read once; mean, then the variance about it, from registers.
template <int NCH>
__device__ __forceinline__ void ln_row_reg(const float* __restrict__ xr, int lane, float eps, float (&v)[NCH][8],
                                           float& mean, float& rstd) {
  constexpr int d = 256 * NCH;
  float s = 0.0f;
#pragma unroll
  for (int c = 0; c < NCH; ++c) {
    const int j = (c * 32 + lane) * 8;
    const float4 a = *reinterpret_cast<const float4*>(xr + j);
    const float4 b = *reinterpret_cast<const float4*>(xr + j + 4);
    v[c][0] = a.x; v[c][1] = a.y; v[c][2] = a.z; v[c][3] = a.w;
    v[c][4] = b.x; v[c][5] = b.y; v[c][6] = b.z; v[c][7] = b.w;
#pragma unroll
    for (int i = 0; i < 8; ++i) s += v[c][i];
  }
  mean = warp_sum(s) / static_cast<float>(d);
  float q = 0.0f;
#pragma unroll
  for (int c = 0; c < NCH; ++c)
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const float a = v[c][i] - mean;
      q = fmaf(a, a, q);
    }
  rstd = rsqrtf(warp_sum(q) / static_cast<float>(d) + eps);
}

// 8 consecutive parameters at element j (bf16 or fp32; 16-byte aligned)
__device__ __forceinline__ void ldw8(const void* w, int bf, int j, float (&o)[8]) {
  if (bf) {
    const uint4 raw = *reinterpret_cast<const uint4*>(static_cast<const bf16*>(w) + j);
    const __nv_bfloat162* p2 = reinterpret_cast<const __nv_bfloat162*>(&raw);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float2 f = __bfloat1622float2(p2[q]);
      o[2 * q] = f.x;
      o[2 * q + 1] = f.y;
    }
  } else {
    const float4 a = *reinterpret_cast<const float4*>(static_cast<const float*>(w) + j);
    const float4 b = *reinterpret_cast<const float4*>(static_cast<const float*>(w) + j + 4);
    o[0] = a.x; o[1] = a.y; o[2] = a.z; o[3] = a.w;
    o[4] = b.x; o[5] = b.y; o[6] = b.z; o[7] = b.w;
  }
}

// 8 consecutive activations at element i (16-byte aligned)
template <class T>
__device__ __forceinline__ void store8(void* out, size_t i, const float (&y)[8]);
template <>
__device__ __forceinline__ void store8<float>(void* out, size_t i, const float (&y)[8]) {
  float4* p = reinterpret_cast<float4*>(static_cast<float*>(out) + i);
  p[0] = make_float4(y[0], y[1], y[2], y[3]);
  p[1] = make_float4(y[4], y[5], y[6], y[7]);
}
template <>
__device__ __forceinline__ void store8<bf16>(void* out, size_t i, const float (&y)[8]) {
  uint32_t pk[4];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    __nv_bfloat162 t = __floats2bfloat162_rn(y[2 * q], y[2 * q + 1]);
    pk[q] = *reinterpret_cast<uint32_t*>(&t);
  }
  *reinterpret_cast<uint4*>(static_cast<bf16*>(out) + i) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
}

// ln_pair_kernel for d = 256 NCH with the row in registers
template <class T, int NCH>
__global__ void __launch_bounds__(WPB * 32) ln_pair_reg_kernel(const float* __restrict__ c, const float* __restrict__ h,
                                                               int M, const void* wc, const void* bc, const void* wh,
                                                               const void* bh, int w_bf16, float eps,
                                                               void* __restrict__ u) {
  pdl_enter();
  constexpr int d = 256 * NCH;
  const int m = blockIdx.x * WPB + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (m >= M) return;
#pragma unroll
  for (int part = 0; part < 2; ++part) {
    const float* xr = (part ? h : c) + static_cast<size_t>(m) * d;
    const void* w = part ? wh : wc;
    const void* b = part ? bh : bc;
    float v[NCH][8], mean, rstd;
    ln_row_reg<NCH>(xr, lane, eps, v, mean, rstd);
#pragma unroll
    for (int ch = 0; ch < NCH; ++ch) {
      const int j = (ch * 32 + lane) * 8;
      float wv[8], bv[8], y[8];
      ldw8(w, w_bf16, j, wv);
      ldw8(b, w_bf16, j, bv);
#pragma unroll
      for (int i = 0; i < 8; ++i) y[i] = (v[ch][i] - mean) * rstd * wv[i] + bv[i];
      store8<T>(u, static_cast<size_t>(m) * 2 * d + part * d + j, y);
    }
  }
}

// layernorm_kernel for d = 256 NCH with the row in registers
template <int NCH>
__global__ void __launch_bounds__(WPB * 32) layernorm_reg_kernel(const float* __restrict__ x, int M, const void* w,
                                                                 const void* b, int w_bf16, float eps,
                                                                 float* __restrict__ out) {
  pdl_enter();
  constexpr int d = 256 * NCH;
  const int m = blockIdx.x * WPB + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (m >= M) return;
  float v[NCH][8], mean, rstd;
  ln_row_reg<NCH>(x + static_cast<size_t>(m) * d, lane, eps, v, mean, rstd);
#pragma unroll
  for (int ch = 0; ch < NCH; ++ch) {
    const int j = (ch * 32 + lane) * 8;
    float wv[8], bv[8], y[8];
    ldw8(w, w_bf16, j, wv);
    ldw8(b, w_bf16, j, bv);
#pragma unroll
    for (int i = 0; i < 8; ++i) y[i] = (v[ch][i] - mean) * rstd * wv[i] + bv[i];
    store8<float>(out, static_cast<size_t>(m) * d + j, y);
  }
}

__global__ void layernorm_kernel(const float* __restrict__ x, int M, int d, const void* w, const void* b, int w_bf16,
                                 float eps, float* __restrict__ out) {
  pdl_enter();
  const int m = blockIdx.x * WPB + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (m >= M) return;
  const float* xr = x + static_cast<size_t>(m) * d;
  float mean, rstd;
  row_mean_var(xr, d, lane, mean, rstd, eps);
  for (int j = lane; j < d; j += 32)
    out[static_cast<size_t>(m) * d + j] = (xr[j] - mean) * rstd * ldw(w, w_bf16, j) + ldw(b, w_bf16, j);
}

// Sandwich norm of a Gemma-3 layer (one warp per row): x += RMSNorm(y) * g_post;
// with g_next also out = RMSNorm(x) * g_next, the pre-norm of the next
// sub-block, from the row just written (read back through L1/L2).
template <class T>
__global__ void post_norm_add_kernel(float* __restrict__ x, const float* __restrict__ y, int M, int d,
                                     const void* __restrict__ g_post, const void* __restrict__ g_next, int w_bf16,
                                     float eps, void* __restrict__ out) {
  pdl_enter();
  const int m = blockIdx.x * WPB + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (m >= M) return;
  float* xr = x + static_cast<size_t>(m) * d;
  const float* yr = y + static_cast<size_t>(m) * d;
  float ss = 0.0f;
  for (int j = lane * 4; j < d; j += 128) {
    const float4 v = *reinterpret_cast<const float4*>(yr + j);
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
  const float inv = rsqrtf(warp_sum(ss) / static_cast<float>(d) + eps);
  float sx = 0.0f;
  for (int j = lane * 4; j < d; j += 128) {
    const float4 v = *reinterpret_cast<const float4*>(yr + j);
    float4 a = *reinterpret_cast<const float4*>(xr + j);
    a.x = fmaf(v.x * inv, ldw(g_post, w_bf16, j + 0), a.x);
    a.y = fmaf(v.y * inv, ldw(g_post, w_bf16, j + 1), a.y);
    a.z = fmaf(v.z * inv, ldw(g_post, w_bf16, j + 2), a.z);
    a.w = fmaf(v.w * inv, ldw(g_post, w_bf16, j + 3), a.w);
    *reinterpret_cast<float4*>(xr + j) = a;
    sx += a.x * a.x + a.y * a.y + a.z * a.z + a.w * a.w;
  }
  if (!g_next) return;
  const float inx = rsqrtf(warp_sum(sx) / static_cast<float>(d) + eps);
  __syncwarp();
  for (int j = lane * 4; j < d; j += 128) {
    const float4 a = *reinterpret_cast<const float4*>(xr + j);
    const size_t o = static_cast<size_t>(m) * d + j;
    store_act<T>(out, o + 0, a.x * inx * ldw(g_next, w_bf16, j + 0));
    store_act<T>(out, o + 1, a.y * inx * ldw(g_next, w_bf16, j + 1));
    store_act<T>(out, o + 2, a.z * inx * ldw(g_next, w_bf16, j + 2));
    store_act<T>(out, o + 3, a.w * inx * ldw(g_next, w_bf16, j + 3));
  }
}

// The same with one 256-thread block per row, for few rows of a wide model
// (a block step of the post-train backbone: 256 rows of 5376).
template <class T>
__global__ void __launch_bounds__(256) post_norm_add_block_kernel(float* __restrict__ x, const float* __restrict__ y,
                                                                  int d, const void* __restrict__ g_post,
                                                                  const void* __restrict__ g_next, int w_bf16,
                                                                  float eps, void* __restrict__ out) {
  pdl_enter();
  __shared__ float red[2][8];
  const int m = blockIdx.x, lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  float* xr = x + static_cast<size_t>(m) * d;
  const float* yr = y + static_cast<size_t>(m) * d;
  float ss = 0.0f;
  for (int j = threadIdx.x * 4; j < d; j += 1024) {
    const float4 v = *reinterpret_cast<const float4*>(yr + j);
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
  ss = warp_sum(ss);
  if (lane == 0) red[0][w] = ss;
  __syncthreads();
  float tot = 0.0f;
#pragma unroll
  for (int k = 0; k < 8; ++k) tot += red[0][k];
  const float inv = rsqrtf(tot / static_cast<float>(d) + eps);
  float sx = 0.0f;
  for (int j = threadIdx.x * 4; j < d; j += 1024) {
    const float4 v = *reinterpret_cast<const float4*>(yr + j);
    float4 a = *reinterpret_cast<const float4*>(xr + j);
    a.x = fmaf(v.x * inv, ldw(g_post, w_bf16, j + 0), a.x);
    a.y = fmaf(v.y * inv, ldw(g_post, w_bf16, j + 1), a.y);
    a.z = fmaf(v.z * inv, ldw(g_post, w_bf16, j + 2), a.z);
    a.w = fmaf(v.w * inv, ldw(g_post, w_bf16, j + 3), a.w);
    *reinterpret_cast<float4*>(xr + j) = a;
    sx += a.x * a.x + a.y * a.y + a.z * a.z + a.w * a.w;
  }
  if (!g_next) return;
  sx = warp_sum(sx);
  if (lane == 0) red[1][w] = sx;
  __syncthreads();   // also orders this block's x writes before the reads below
  float totx = 0.0f;
#pragma unroll
  for (int k = 0; k < 8; ++k) totx += red[1][k];
  const float inx = rsqrtf(totx / static_cast<float>(d) + eps);
  for (int j = threadIdx.x * 4; j < d; j += 1024) {
    const float4 a = *reinterpret_cast<const float4*>(xr + j);
    const size_t o = static_cast<size_t>(m) * d + j;
    store_act<T>(out, o + 0, a.x * inx * ldw(g_next, w_bf16, j + 0));
    store_act<T>(out, o + 1, a.y * inx * ldw(g_next, w_bf16, j + 1));
    store_act<T>(out, o + 2, a.z * inx * ldw(g_next, w_bf16, j + 2));
    store_act<T>(out, o + 3, a.w * inx * ldw(g_next, w_bf16, j + 3));
  }
}

__global__ void rms_scale_kernel(const float* __restrict__ x, int M, int d, float eps, float* __restrict__ s) {
  pdl_enter();
  const int m = blockIdx.x * WPB + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (m >= M) return;
  const float* xr = x + static_cast<size_t>(m) * d;
  float ss = 0.0f;
  for (int j = lane; j < d; j += 32) ss += xr[j] * xr[j];
  ss = warp_sum(ss);
  if (lane == 0) s[m] = sqrtf(ss / static_cast<float>(d) + eps);
}

// out = x / s[row], element-wise over four columns per thread (d % 4 == 0)
template <class T>
__global__ void scale_rows_kernel(const float* __restrict__ x, const float* __restrict__ sc, int M, int d,
                                  void* __restrict__ out) {
  pdl_enter();
  const size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x;
  if (i >= static_cast<size_t>(M) * (d / 4)) return;
  const size_t e = i * 4;
  const float s = sc[e / d];
  const float4 v = *reinterpret_cast<const float4*>(x + e);
  store_act<T>(out, e + 0, v.x / s);
  store_act<T>(out, e + 1, v.y / s);
  store_act<T>(out, e + 2, v.z / s);
  store_act<T>(out, e + 3, v.w / s);
}

// s[row] = sqrt(mean(x^2) + eps), one 256-thread block per row (few rows)
__global__ void __launch_bounds__(256) rms_scale_block_kernel(const float* __restrict__ x, int d, float eps,
                                                              float* __restrict__ s) {
  pdl_enter();
  __shared__ float red[8];
  const int m = blockIdx.x;
  const float* xr = x + static_cast<size_t>(m) * d;
  float ss = 0.0f;
  for (int j = threadIdx.x; j < d; j += 256) ss += xr[j] * xr[j];
  ss = warp_sum(ss);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  if (threadIdx.x == 0) {
    float tot = 0.0f;
    for (int w = 0; w < 8; ++w) tot += red[w];
    s[m] = sqrtf(tot / static_cast<float>(d) + eps);
  }
}

struct Parts {
  const float* p[4];
  int w[4];
  int n;
};

// out[m] = [parts[0][m], parts[1][m], ...], one output element per thread
template <class T>
__global__ void concat_kernel(Parts parts, int M, int width, void* __restrict__ out) {
  pdl_enter();
  const size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x;
  if (i >= static_cast<size_t>(M) * width) return;
  const int m = static_cast<int>(i / width);
  int col = static_cast<int>(i % width), k = 0;
  while (col >= parts.w[k]) col -= parts.w[k++];
  store_act<T>(out, i, parts.p[k][static_cast<size_t>(m) * parts.w[k] + col]);
}

__global__ void sub_kernel(const float* __restrict__ a, const float* __restrict__ b, size_t n, float* __restrict__ o) {
  pdl_enter();
  for (size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<size_t>(gridDim.x) * blockDim.x)
    o[i] = a[i] - b[i];
}

// tab[j][pos] = (cos, sin)(pos * theta^(-2j/hd)), angles evaluated in double
__global__ void rope_table_kernel(float2* tab, int n_pos, int half, int hd, double theta) {
  pdl_enter();
  const size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x;
  if (i >= static_cast<size_t>(n_pos) * half) return;
  const int j = static_cast<int>(i / n_pos), pos = static_cast<int>(i % n_pos);
  const double inv = pow(theta, -2.0 * j / hd);
  const double ang = static_cast<double>(pos) * inv;
  tab[i] = make_float2(static_cast<float>(cos(ang)), static_cast<float>(sin(ang)));
}

__global__ void fill_canvas_kernel(int32_t* z, int ldz, const int32_t* prompt, int batch, int P, int total,
                                   int mask_id) {
  pdl_enter();
  const size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x;
  if (i >= static_cast<size_t>(batch) * total) return;
  const int b = static_cast<int>(i / total), p = static_cast<int>(i % total);
  z[static_cast<size_t>(b) * ldz + p] = p < P ? prompt[static_cast<size_t>(b) * P + p] : mask_id;
}

__global__ void copy_i32_kernel(const int32_t* src, int lds, int32_t* dst, int ldd, int batch, int cols) {
  pdl_enter();
  const size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x;
  if (i >= static_cast<size_t>(batch) * cols) return;
  const int b = static_cast<int>(i / cols), c = static_cast<int>(i % cols);
  dst[static_cast<size_t>(b) * ldd + c] = src[static_cast<size_t>(b) * lds + c];
}

inline dim3 rows_grid(int M) { return dim3((M + WPB - 1) / WPB); }
inline const char* err() {
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? nullptr : cudaGetErrorString(e);
}
}  // namespace

const char* embed_rows(const int32_t* z, int ldz, int batch, int rows, const void* E, int e_bf16, int d, int vocab,
                       float* out, float* out2, cudaStream_t s, const float* add, int add_first,
                       const float* add_div) {
  const int M = batch * rows;
  if (M <= 0) return nullptr;
  if (d % 4) return "d_model must be a multiple of 4";
  if (add && (add_first < 0 || add_first > rows)) return "self-conditioning rows out of range";
  launch_pdl(embed_kernel, rows_grid(M), WPB * 32, 0, s, z, ldz, rows, M, E, e_bf16, d, vocab, out, out2, add,
             add_first, add_div);
  return err();
}

const char* rmsnorm_rows(const float* x, int M, int d, const void* gain, int w_bf16, float eps, void* out, int ldo,
                         int act_bf16, cudaStream_t s, const int32_t* rows_idx, int lo_off) {
  if (M <= 0) return nullptr;
  if (!act_bf16) lo_off = 0;       // fp32 activations are not split
  if (lo_off > 0 && (lo_off < d || lo_off + d > ldo)) return "split operand: the remainder columns must follow the row";
  if (M < 1024) {   // few rows: a block per row keeps enough SMs busy
    if (act_bf16)
      launch_pdl(rmsnorm_block_kernel<bf16>, M, 256, 0, s, x, d, gain, w_bf16, eps, out, ldo, rows_idx, lo_off);
    else
      launch_pdl(rmsnorm_block_kernel<float>, M, 256, 0, s, x, d, gain, w_bf16, eps, out, ldo, rows_idx, lo_off);
    return err();
  }
  const bool vec = act_bf16 && w_bf16 && ldo % 8 == 0 && lo_off % 8 == 0 &&
                   ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(out) | reinterpret_cast<uintptr_t>(gain)) & 15) == 0;
  if (vec) {
    const bf16* g = static_cast<const bf16*>(gain);
    bf16* o = static_cast<bf16*>(out);
    switch (d) {
      case 256: launch_pdl(rmsnorm_reg_kernel<1>, rows_grid(M), WPB * 32, 0, s, x, M, g, eps, o, ldo, rows_idx, lo_off); return err();
      case 512: launch_pdl(rmsnorm_reg_kernel<2>, rows_grid(M), WPB * 32, 0, s, x, M, g, eps, o, ldo, rows_idx, lo_off); return err();
      case 768: launch_pdl(rmsnorm_reg_kernel<3>, rows_grid(M), WPB * 32, 0, s, x, M, g, eps, o, ldo, rows_idx, lo_off); return err();
      case 1024: launch_pdl(rmsnorm_reg_kernel<4>, rows_grid(M), WPB * 32, 0, s, x, M, g, eps, o, ldo, rows_idx, lo_off); return err();
      case 2048: launch_pdl(rmsnorm_reg_kernel<8>, rows_grid(M), WPB * 32, 0, s, x, M, g, eps, o, ldo, rows_idx, lo_off); return err();
      default: break;
    }
  }
  if (act_bf16)
    launch_pdl(rmsnorm_kernel<bf16>, rows_grid(M), WPB * 32, 0, s, x, M, d, gain, w_bf16, eps, out, ldo, rows_idx, lo_off);
  else
    launch_pdl(rmsnorm_kernel<float>, rows_grid(M), WPB * 32, 0, s, x, M, d, gain, w_bf16, eps, out, ldo, rows_idx, lo_off);
  return err();
}

// true when every pointer is 16-byte aligned (the register kernels' vector accesses)
static bool all16(std::initializer_list<const void*> ps) {
  for (const void* p : ps)
    if (reinterpret_cast<uintptr_t>(p) & 15) return false;
  return true;
}

template <class T>
static bool ln_pair_reg(const float* c, const float* h, int M, int d, const void* wc, const void* bc, const void* wh,
                 const void* bh, int w_bf16, float eps, void* u, cudaStream_t s) {
  switch (d) {
    case 256: launch_pdl(ln_pair_reg_kernel<T, 1>, rows_grid(M), WPB * 32, 0, s, c, h, M, wc, bc, wh, bh, w_bf16, eps, u); return true;
    case 512: launch_pdl(ln_pair_reg_kernel<T, 2>, rows_grid(M), WPB * 32, 0, s, c, h, M, wc, bc, wh, bh, w_bf16, eps, u); return true;
    case 768: launch_pdl(ln_pair_reg_kernel<T, 3>, rows_grid(M), WPB * 32, 0, s, c, h, M, wc, bc, wh, bh, w_bf16, eps, u); return true;
    case 1024: launch_pdl(ln_pair_reg_kernel<T, 4>, rows_grid(M), WPB * 32, 0, s, c, h, M, wc, bc, wh, bh, w_bf16, eps, u); return true;
    case 2048: launch_pdl(ln_pair_reg_kernel<T, 8>, rows_grid(M), WPB * 32, 0, s, c, h, M, wc, bc, wh, bh, w_bf16, eps, u); return true;
    default: return false;
  }
}

const char* ln_pair_rows(const float* c, const float* h, int M, int d, const void* wc, const void* bc, const void* wh,
                         const void* bh, int w_bf16, float eps, void* u, int act_bf16, cudaStream_t s) {
  if (M <= 0) return nullptr;
  if (all16({c, h, wc, bc, wh, bh, u})) {
    const bool done = act_bf16 ? ln_pair_reg<bf16>(c, h, M, d, wc, bc, wh, bh, w_bf16, eps, u, s)
                               : ln_pair_reg<float>(c, h, M, d, wc, bc, wh, bh, w_bf16, eps, u, s);
    if (done) return err();
  }
  if (act_bf16)
    launch_pdl(ln_pair_kernel<bf16>, rows_grid(M), WPB * 32, 0, s, c, h, M, d, wc, bc, wh, bh, w_bf16, eps, u);
  else
    launch_pdl(ln_pair_kernel<float>, rows_grid(M), WPB * 32, 0, s, c, h, M, d, wc, bc, wh, bh, w_bf16, eps, u);
  return err();
}

const char* layernorm_rows(const float* x, int M, int d, const void* w, const void* b, int w_bf16, float eps,
                           float* out, cudaStream_t s) {
  if (M <= 0) return nullptr;
  if (all16({x, w, b, out})) {
    switch (d) {
      case 256: launch_pdl(layernorm_reg_kernel<1>, rows_grid(M), WPB * 32, 0, s, x, M, w, b, w_bf16, eps, out); return err();
      case 512: launch_pdl(layernorm_reg_kernel<2>, rows_grid(M), WPB * 32, 0, s, x, M, w, b, w_bf16, eps, out); return err();
      case 768: launch_pdl(layernorm_reg_kernel<3>, rows_grid(M), WPB * 32, 0, s, x, M, w, b, w_bf16, eps, out); return err();
      case 1024: launch_pdl(layernorm_reg_kernel<4>, rows_grid(M), WPB * 32, 0, s, x, M, w, b, w_bf16, eps, out); return err();
      case 2048: launch_pdl(layernorm_reg_kernel<8>, rows_grid(M), WPB * 32, 0, s, x, M, w, b, w_bf16, eps, out); return err();
      default: break;
    }
  }
  launch_pdl(layernorm_kernel, rows_grid(M), WPB * 32, 0, s, x, M, d, w, b, w_bf16, eps, out);
  return err();
}

const char* rms_scale_rows(const float* x, int M, int d, float eps, float* s_out, cudaStream_t st) {
  if (M <= 0) return nullptr;
  if (M < 1024) {   // few rows: a block per row keeps enough SMs busy
    launch_pdl(rms_scale_block_kernel, M, 256, 0, st, x, d, eps, s_out);
    return err();
  }
  launch_pdl(rms_scale_kernel, rows_grid(M), WPB * 32, 0, st, x, M, d, eps, s_out);
  return err();
}

const char* post_norm_add(float* x, const float* y, int M, int d, const void* g_post, const void* g_next, int w_bf16,
                          float eps, void* out, int act_bf16, cudaStream_t s) {
  if (M <= 0) return nullptr;
  if (d % 4) return "post-norm rows need d % 4 == 0";
  if (M < 1024) {   // few rows: a block per row keeps enough SMs busy
    if (act_bf16)
      launch_pdl(post_norm_add_block_kernel<bf16>, M, 256, 0, s, x, y, d, g_post, g_next, w_bf16, eps, out);
    else
      launch_pdl(post_norm_add_block_kernel<float>, M, 256, 0, s, x, y, d, g_post, g_next, w_bf16, eps, out);
    return err();
  }
  if (act_bf16)
    launch_pdl(post_norm_add_kernel<bf16>, rows_grid(M), WPB * 32, 0, s, x, y, M, d, g_post, g_next, w_bf16, eps, out);
  else
    launch_pdl(post_norm_add_kernel<float>, rows_grid(M), WPB * 32, 0, s, x, y, M, d, g_post, g_next, w_bf16, eps,
               out);
  return err();
}

const char* scale_rows(const float* x, const float* sc, int M, int d, void* out, int act_bf16, cudaStream_t s) {
  if (M <= 0) return nullptr;
  if (d % 4) return "scale_rows needs d % 4 == 0";
  const unsigned blocks = static_cast<unsigned>((static_cast<size_t>(M) * (d / 4) + 255) / 256);
  if (act_bf16)
    launch_pdl(scale_rows_kernel<bf16>, blocks, 256, 0, s, x, sc, M, d, out);
  else
    launch_pdl(scale_rows_kernel<float>, blocks, 256, 0, s, x, sc, M, d, out);
  return err();
}

const char* concat_rows(const float* const* parts, const int* widths, int n_parts, int M, void* out, int act_bf16,
                        cudaStream_t s) {
  if (M <= 0) return nullptr;
  if (n_parts < 1 || n_parts > 4) return "concat of 1..4 parts";
  Parts p{};
  int width = 0;
  for (int i = 0; i < n_parts; ++i) {
    p.p[i] = parts[i];
    p.w[i] = widths[i];
    width += widths[i];
  }
  p.n = n_parts;
  const unsigned blocks = static_cast<unsigned>((static_cast<size_t>(M) * width + 255) / 256);
  if (act_bf16)
    launch_pdl(concat_kernel<bf16>, blocks, 256, 0, s, p, M, width, out);
  else
    launch_pdl(concat_kernel<float>, blocks, 256, 0, s, p, M, width, out);
  return err();
}

const char* sub_rows(const float* a, const float* b, int M, int d, float* out, cudaStream_t s) {
  const size_t n = static_cast<size_t>(M) * d;
  if (n == 0) return nullptr;
  const int blocks = static_cast<int>((n + 255) / 256 < 65535 ? (n + 255) / 256 : 65535);
  launch_pdl(sub_kernel, blocks, 256, 0, s, a, b, n, out);
  return err();
}

const char* rope_table(float2* tab, int n_pos, int head_dim, float theta, cudaStream_t s) {
  const size_t n = static_cast<size_t>(n_pos) * (head_dim / 2);
  if (n == 0) return nullptr;
  launch_pdl(rope_table_kernel, static_cast<unsigned>((n + 255) / 256), 256, 0, s, tab, n_pos, head_dim / 2, head_dim,
                                                                            static_cast<double>(theta));
  return err();
}

const char* fill_canvas(int32_t* z, int ldz, const int32_t* prompt, int batch, int prompt_len, int total,
                        int mask_id, cudaStream_t s) {
  const size_t n = static_cast<size_t>(batch) * total;
  if (n == 0) return nullptr;
  launch_pdl(fill_canvas_kernel, static_cast<unsigned>((n + 255) / 256), 256, 0, s, z, ldz, prompt, batch, prompt_len,
                                                                             total, mask_id);
  return err();
}

const char* copy_rows_i32(const int32_t* src, int lds, int32_t* dst, int ldd, int batch, int cols, cudaStream_t s) {
  const size_t n = static_cast<size_t>(batch) * cols;
  if (n == 0) return nullptr;
  launch_pdl(copy_i32_kernel, static_cast<unsigned>((n + 255) / 256), 256, 0, s, src, lds, dst, ldd, batch, cols);
  return err();
}

}  // namespace tadm
