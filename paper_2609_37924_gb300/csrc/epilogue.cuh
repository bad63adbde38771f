// GEMM epilogues.  Every GEMM of the path computes acc = A B^T for one output
// row at a time and hands the accumulator row, in chunks of 32 fp32 columns,
// to one of these functions.  They fuse what follows each projection: the
// residual add, RoPE and the K/V cache write, the GLU activation, the two
// fusion-module epilogues (gate / hidden activations; h + g * Delta), and the
// per-row partial max / argmax / sum-exp of the output head.
#pragma once
#include "common.cuh"

namespace tadm {

enum EpiKind : int {
  EPI_STORE = 0,     // out = acc
  EPI_RESID = 1,     // resid += acc (+ bias)
  EPI_QKV = 2,       // split into Q / K / V heads, optional QK-norm and RoPE, K and V^T into the cache
  EPI_GLU = 3,       // out = act(gate) * up (gate and up are the two halves of the tile)
  EPI_FUSION1 = 4,   // [g | hidden] = [sigmoid(acc + b) | GELU(acc + b)]
  EPI_FUSION2 = 5,   // out = h + g * (acc + b)
  EPI_LMHEAD = 6,    // per-row (max, sum exp, argmax) partial of this column tile
  EPI_PA_UP = 7,     // out = H0 + g[row] * sH[row] * acc
  EPI_SILU = 8,      // out = SiLU(acc)
  EPI_ADD = 9,       // out = base + acc (+ act copy in out2)
  EPI_PA_GATE = 10,  // g[row] = sigmoid(sum_j SiLU(acc_j) w_j + b), single column tile
};

struct EpiParams {
  int M, N;                 // output rows / columns (EPI_GLU: the F output columns)
  void* out;
  int ldo, out_bf16;        // out element type: bf16 (1) or fp32 (0)
  float* resid;
  int ldr;
  int resid_tma;            // EPI_RESID on the tensor-core path: resid += acc by TMA reduce-add (map in the source)
  const float* base;        // EPI_ADD base, EPI_FUSION2 h, EPI_PA_UP H0
  int ldb;
  const void* bias;         // [N] weights dtype
  int bias_bf16;
  // EPI_QKV: q [B, Hq, R, hd], k [B, Hkv, kv_stride, hd], v transposed [B, Hkv, hd, kv_stride]
  void *q, *k, *v;
  int R, ctx, kv_stride, n_heads, n_kv_heads, head_dim, rope;
  const float2* rope_tab;   // [head_dim / 2][n_pos] = (cos, sin): a warp's consecutive positions read consecutive entries
  int rope_npos;
  // EPI_QKV with QK-norm (Gemma-3 layers): RMSNorm over head_dim of every Q / K head before RoPE,
  // gains [head_dim] in the weights' type (bias_bf16); null: no QK-norm
  const void *q_gain, *k_gain;
  float qk_eps;
  // EPI_GLU
  int glu;                  // 0 SiLU, 1 tanh-GELU
  // EPI_FUSION1 / EPI_ADD
  int d_split;
  void* out2;
  int ldo2;
  // EPI_FUSION2 (act type [M, N]) / EPI_PA_UP (fp32 [M])
  const void* gate;
  int ldg;
  const float* rowscale;
  // EPI_LMHEAD
  float* part;              // [M][n_tiles][3] = (max, sum, argmax bits)
  int n_tiles, mask_id;
  float* logits;            // optional fp32 [M, ld_logits]
  int ld_logits;
  // EPI_PA_GATE: vec = W_g2 [N] (weights dtype), bias = b_g [1]
  const void* vec;
};

__device__ __forceinline__ float ld_param(const void* p, int bf, int i) {
  return bf ? __bfloat162float(static_cast<const bf16*>(p)[i]) : static_cast<const float*>(p)[i];
}

// Activations of the epilogues.  Their outputs feed bf16 GEMM operands (or
// are rounded to bf16), so they use the fast exp2-based exponential and the
// approximate reciprocal / division, whose errors (a few fp32 ulp) lie far
// below bf16's rounding step.  At the extremes: exp overflow gives
// x / inf = -0 for SiLU and 0 for the sigmoid, exp underflow gives x and 1.
__device__ __forceinline__ float silu_f(float x) { return __fdividef(x, 1.0f + __expf(-x)); }
__device__ __forceinline__ float sigmoid_f(float x) { return __fdividef(1.0f, 1.0f + __expf(-x)); }
// erf by the rational approximation of Abramowitz & Stegun, Handbook of
// Mathematical Functions (1964), formula 7.1.26 (after Hastings):
//   erf(z) = 1 - (a1 t + a2 t^2 + a3 t^3 + a4 t^4 + a5 t^5) exp(-z^2),
//   t = 1 / (1 + p z), z >= 0, |error| <= 1.5e-7; erf is odd.
__device__ __forceinline__ float erf_as7126(float x) {
  const float z = fabsf(x);
  const float t = __fdividef(1.0f, fmaf(0.3275911f, z, 1.0f));
  const float poly =
      t * fmaf(fmaf(fmaf(fmaf(1.061405429f, t, -1.453152027f), t, 1.421413741f), t, -0.284496736f), t, 0.254829592f);
  return copysignf(fmaf(-poly, __expf(-z * z), 1.0f), x);
}
__device__ __forceinline__ float gelu_erf_f(float x) { return 0.5f * x * (1.0f + erf_as7126(x * 0.70710678118654752f)); }
// tanh(y) = 1 - 2 / (1 + exp(2y)): +-1 at the extremes, absolute error ~1e-7 near 0
__device__ __forceinline__ float tanh_fast(float y) { return 1.0f - __fdividef(2.0f, 1.0f + __expf(2.0f * y)); }
__device__ __forceinline__ float gelu_tanh_f(float x) {
  return 0.5f * x * (1.0f + tanh_fast(0.79788456080286536f * (x + 0.044715f * x * x * x)));
}

// Stores 32 consecutive values (n0 .. n0+31) of one row; `n_valid` of them.
__device__ __forceinline__ void store32(void* base, int bf, size_t off, const float (&v)[32], int n_valid) {
  if (bf) {
    bf16* p = static_cast<bf16*>(base) + off;
    if (n_valid >= 32 && (off & 7) == 0) {
      uint4* p4 = reinterpret_cast<uint4*>(p);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        __nv_bfloat162 t0 = __floats2bfloat162_rn(v[8 * i + 0], v[8 * i + 1]);
        __nv_bfloat162 t1 = __floats2bfloat162_rn(v[8 * i + 2], v[8 * i + 3]);
        __nv_bfloat162 t2 = __floats2bfloat162_rn(v[8 * i + 4], v[8 * i + 5]);
        __nv_bfloat162 t3 = __floats2bfloat162_rn(v[8 * i + 6], v[8 * i + 7]);
        uint4 u;
        u.x = *reinterpret_cast<uint32_t*>(&t0);
        u.y = *reinterpret_cast<uint32_t*>(&t1);
        u.z = *reinterpret_cast<uint32_t*>(&t2);
        u.w = *reinterpret_cast<uint32_t*>(&t3);
        p4[i] = u;
      }
    } else {
      for (int i = 0; i < n_valid; ++i) p[i] = __float2bfloat16_rn(v[i]);
    }
  } else {
    float* p = static_cast<float*>(base) + off;
    if (n_valid >= 32 && (off & 3) == 0) {
      float4* p4 = reinterpret_cast<float4*>(p);
#pragma unroll
      for (int i = 0; i < 8; ++i) p4[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
    } else {
      for (int i = 0; i < n_valid; ++i) p[i] = v[i];
    }
  }
}

// Stores 32 values of one row as one column of a transposed layout: element i
// goes to base[off + i * stride].  Across a warp whose lanes hold consecutive
// rows, each of the 32 stores writes 32 consecutive elements.
__device__ __forceinline__ void store_col32(void* base, int bf, size_t off, int stride, const float (&v)[32]) {
  if (bf) {
    bf16* p = static_cast<bf16*>(base) + off;
#pragma unroll
    for (int i = 0; i < 32; ++i) p[static_cast<size_t>(i) * stride] = __float2bfloat16_rn(v[i]);
  } else {
    float* p = static_cast<float*>(base) + off;
#pragma unroll
    for (int i = 0; i < 32; ++i) p[static_cast<size_t>(i) * stride] = v[i];
  }
}

__device__ __forceinline__ void load32f(const float* p, int n_valid, float (&v)[32]) {
  if (n_valid >= 32 && (reinterpret_cast<uintptr_t>(p) & 15) == 0) {
    const float4* p4 = reinterpret_cast<const float4*>(p);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      float4 t = p4[i];
      v[4 * i] = t.x; v[4 * i + 1] = t.y; v[4 * i + 2] = t.z; v[4 * i + 3] = t.w;
    }
  } else {
    for (int i = 0; i < 32; ++i) v[i] = i < n_valid ? p[i] : 0.0f;
  }
}

__device__ __forceinline__ void load32a(const void* p, int bf, size_t off, int n_valid, float (&v)[32]) {
  if (bf) {
    const bf16* q = static_cast<const bf16*>(p) + off;
    for (int i = 0; i < 32; ++i) v[i] = i < n_valid ? __bfloat162float(q[i]) : 0.0f;
  } else {
    load32f(static_cast<const float*>(p) + off, n_valid, v);
  }
}

// One output row of one column tile.  `ncols` accumulator columns (a multiple
// of 64) are available from src.load(chunk, v); the tile's first output column
// is n_blk * ncols (n_blk * ncols / 2 for EPI_GLU).  Control flow is uniform
// across a warp except for the stores (src.load may be warp-collective).
//
// The tile's columns may be split between `nsplit` threads per row (one per
// warp of a lane quadrant); split `part` handles its share: chunks
// [part * nch / nsplit, (part + 1) * nch / nsplit) (for EPI_GLU the same share
// of gate chunks and their up partners; for EPI_QKV whole heads; EPI_LMHEAD
// writes one partial per split, indexed n_blk * nsplit + part; EPI_PA_GATE
// needs nsplit == 1).
template <int EPI, class Src>
__device__ __forceinline__ void epilogue_row(const EpiParams& p, int m, int n_blk, int ncols, Src& src,
                                             int part = 0, int nsplit = 1) {
  const bool row_ok = m < p.M;
  const int nch = ncols / 32;
  const int c_lo = part * nch / nsplit, c_hi = (part + 1) * nch / nsplit;
  float v[32];
  // Sources that can stage (tensor-core path) write bf16 outputs 64 columns at
  // a time through shared memory with one TMA store per warp (full lines).
  if constexpr (Src::kStaged && (EPI == EPI_STORE || EPI == EPI_FUSION1)) {
    if (src.staged()) {
      float w[32];
      for (int c = c_lo; c + 1 < c_hi; c += 2) {
        src.load(c, v);
        src.load(c + 1, w);
        const int n0 = n_blk * ncols + 32 * c;
        int which = 0, x = n0;
        if constexpr (EPI == EPI_FUSION1) {
          // one bias value per lane, broadcast by shuffles; the activation is
          // chosen once per 64 columns (d_split is a multiple of 64)
          const int lane = threadIdx.x & 31;
          const float bl0 = n0 + lane < p.N ? ld_param(p.bias, p.bias_bf16, n0 + lane) : 0.0f;
          const float bl1 = n0 + 32 + lane < p.N ? ld_param(p.bias, p.bias_bf16, n0 + 32 + lane) : 0.0f;
          const bool gate = n0 < p.d_split;
          if (gate) {
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              v[i] = sigmoid_f(v[i] + __shfl_sync(0xffffffffu, bl0, i));
              w[i] = sigmoid_f(w[i] + __shfl_sync(0xffffffffu, bl1, i));
            }
          } else {
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              v[i] = gelu_erf_f(v[i] + __shfl_sync(0xffffffffu, bl0, i));
              w[i] = gelu_erf_f(w[i] + __shfl_sync(0xffffffffu, bl1, i));
            }
          }
          which = gate ? 0 : 1;
          x = gate ? n0 : n0 - p.d_split;
        }
        src.store64(which, x, v, w);
      }
      return;
    }
  }
  // residual add on the tensor-core path: the warp's 32 x 32 chunk (+ bias) goes
  // through its shared-memory box and one TMA reduce-add (resid += chunk at
  // L2), so the epilogue never waits on a load of the residual stream.  Each
  // element receives exactly one add per GEMM: the result is deterministic.
  // The next chunk's TMEM load is issued before this chunk's box wait and
  // reduce, so its latency overlaps them.
  if constexpr (Src::kStaged && EPI == EPI_RESID) {
    if (src.has_box() && p.resid_tma) {
      uint32_t cur[32], nxt[32];
      if (c_lo < c_hi) {
        src.load_async(c_lo, cur);
        src.wait_ld(cur);
      }
      for (int c = c_lo; c < c_hi; ++c) {
        if (c + 1 < c_hi) src.load_async(c + 1, nxt);
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(cur[i]);
        const int n0 = n_blk * ncols + 32 * c;
        if (p.bias) {
          const int lane = threadIdx.x & 31;
          const float bl = n0 + lane < p.N ? ld_param(p.bias, p.bias_bf16, n0 + lane) : 0.0f;
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] += __shfl_sync(0xffffffffu, bl, i);
        }
        if (n0 < p.N && src.row0 < p.M) src.reduce32(n0, v);   // the map clips ragged rows / columns
        if (c + 1 < c_hi) {
          src.wait_ld(nxt);
#pragma unroll
          for (int i = 0; i < 32; ++i) cur[i] = nxt[i];
        }
      }
      return;
    }
  }
  // fp32 read-modify-write epilogues on the tensor-core path: the warp's 32 x 32
  // accumulator chunk is transposed through its shared-memory box so that each
  // global access instruction covers 32 consecutive columns of one row.
  if constexpr (Src::kStaged && (EPI == EPI_RESID || EPI == EPI_FUSION2)) {
    if (src.has_box()) {
      const int lane = threadIdx.x & 31;
      for (int c = c_lo; c < c_hi; ++c) {
        src.load(c, v);
        src.put_row(v);
        const int n = n_blk * ncols + 32 * c + lane;
        const bool col_ok = n < p.N;
        const float bias = (p.bias && col_ok) ? ld_param(p.bias, p.bias_bf16, n) : 0.0f;
        const int nrows = min(32, p.M - src.row0);
#pragma unroll
        for (int h0 = 0; h0 < 32; h0 += 16) {     // 16 rows at a time: loads first, then the stores
          float xv[16], gv[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const size_t m_i = static_cast<size_t>(src.row0 + h0 + i);
            const bool ok = h0 + i < nrows && col_ok;
            if constexpr (EPI == EPI_RESID) {
              xv[i] = ok ? p.resid[m_i * p.ldr + n] : 0.0f;
            } else {
              xv[i] = ok ? p.base[m_i * p.ldb + n] : 0.0f;
              gv[i] = ok ? ld_param(p.gate, p.out_bf16, static_cast<int>(m_i * p.ldg + n)) : 0.0f;
            }
          }
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const size_t m_i = static_cast<size_t>(src.row0 + h0 + i);
            if (h0 + i < nrows && col_ok) {
              const float a = src.get(h0 + i);
              if constexpr (EPI == EPI_RESID) p.resid[m_i * p.ldr + n] = xv[i] + a + bias;
              else static_cast<float*>(p.out)[m_i * p.ldo + n] = xv[i] + gv[i] * (a + bias);
            }
          }
        }
        __syncwarp();   // the box is rewritten by the next chunk
      }
      return;
    }
  }
  if constexpr (EPI == EPI_STORE || EPI == EPI_RESID || EPI == EPI_SILU || EPI == EPI_ADD ||
                EPI == EPI_FUSION1 || EPI == EPI_FUSION2 || EPI == EPI_PA_UP) {
    for (int c = c_lo; c < c_hi; ++c) {
      src.load(c, v);
      const int n0 = n_blk * ncols + 32 * c;
      const int nv = min(32, p.N - n0);
      if (!row_ok || nv <= 0) continue;
      const size_t mrow = static_cast<size_t>(m);
      if constexpr (EPI == EPI_STORE) {
        store32(p.out, p.out_bf16, mrow * p.ldo + n0, v, nv);
      } else if constexpr (EPI == EPI_SILU) {
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] = silu_f(v[i]);
        store32(p.out, p.out_bf16, mrow * p.ldo + n0, v, nv);
      } else if constexpr (EPI == EPI_RESID) {
        float r[32];
        float* rp = p.resid + mrow * p.ldr + n0;
        load32f(rp, nv, r);
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          float b = (p.bias && i < nv) ? ld_param(p.bias, p.bias_bf16, n0 + i) : 0.0f;
          r[i] += v[i] + b;
        }
        store32(p.resid, 0, mrow * p.ldr + n0, r, nv);
      } else if constexpr (EPI == EPI_ADD) {
        float r[32];
        load32f(p.base + mrow * p.ldb + n0, nv, r);
#pragma unroll
        for (int i = 0; i < 32; ++i) r[i] += v[i];
        store32(p.out, 0, mrow * p.ldo + n0, r, nv);
        if (p.out2) store32(p.out2, p.out_bf16, mrow * p.ldo2 + n0, r, nv);
      } else if constexpr (EPI == EPI_FUSION1) {
        float g[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const int n = n0 + i;
          const float b = (i < nv) ? ld_param(p.bias, p.bias_bf16, n) : 0.0f;
          g[i] = (n < p.d_split) ? sigmoid_f(v[i] + b) : gelu_erf_f(v[i] + b);
        }
        // d_split is a multiple of 32: a chunk is all gate or all hidden
        if (n0 < p.d_split)
          store32(p.out, p.out_bf16, mrow * p.ldo + n0, g, min(nv, p.d_split - n0));
        else
          store32(p.out2, p.out_bf16, mrow * p.ldo2 + (n0 - p.d_split), g, nv);
      } else if constexpr (EPI == EPI_FUSION2) {
        float h[32], g[32];
        load32f(p.base + mrow * p.ldb + n0, nv, h);
        load32a(p.gate, p.out_bf16, mrow * p.ldg + n0, nv, g);
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const float b = (p.bias && i < nv) ? ld_param(p.bias, p.bias_bf16, n0 + i) : 0.0f;
          h[i] = h[i] + g[i] * (v[i] + b);
        }
        store32(p.out, 0, mrow * p.ldo + n0, h, nv);
      } else if constexpr (EPI == EPI_PA_UP) {
        float h[32];
        load32f(p.base + mrow * p.ldb + n0, nv, h);
        const float gs = static_cast<const float*>(p.gate)[m] * p.rowscale[m];
#pragma unroll
        for (int i = 0; i < 32; ++i) h[i] = h[i] + gs * v[i];
        store32(p.out, 0, mrow * p.ldo + n0, h, nv);
      }
    }
  } else if constexpr (EPI == EPI_GLU) {
    const int half = ncols / 2;
    const int g_lo = part * (half / 32) / nsplit, g_hi = (part + 1) * (half / 32) / nsplit;
    if constexpr (Src::kStaged) {
      if (src.staged()) {
        float w[32], u[32];
        for (int c = g_lo; c + 1 < g_hi; c += 2) {
          src.load(c, v);
          src.load(c + half / 32, u);
          if (p.glu) {
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = gelu_tanh_f(v[i]) * u[i];
          } else {
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] = silu_f(v[i]) * u[i];
          }
          src.load(c + 1, w);
          src.load(c + 1 + half / 32, u);
          if (p.glu) {
#pragma unroll
            for (int i = 0; i < 32; ++i) w[i] = gelu_tanh_f(w[i]) * u[i];
          } else {
#pragma unroll
            for (int i = 0; i < 32; ++i) w[i] = silu_f(w[i]) * u[i];
          }
          src.store64(0, n_blk * half + 32 * c, v, w);
        }
        return;
      }
    }
    for (int c = g_lo; c < g_hi; ++c) {
      float u[32];
      src.load(c, v);
      src.load(c + half / 32, u);
      const int n0 = n_blk * half + 32 * c;
      const int nv = min(32, p.N - n0);
      if (!row_ok || nv <= 0) continue;
#pragma unroll
      for (int i = 0; i < 32; ++i) v[i] = (p.glu ? gelu_tanh_f(v[i]) : silu_f(v[i])) * u[i];
      store32(p.out, p.out_bf16, static_cast<size_t>(m) * p.ldo + n0, v, nv);
    }
  } else if constexpr (EPI == EPI_QKV) {
    const int hd = p.head_dim;
    const int hpt = ncols / hd;       // heads per tile
    const int b = m / p.R, r = m - (m / p.R) * p.R;
    const int pos = p.ctx + r;
    for (int hh = part * hpt / nsplit; hh < (part + 1) * hpt / nsplit; ++hh) {
      const int nb = n_blk * ncols + hh * hd;
      const int gh = nb / hd;
      int region = 2, head = gh - p.n_heads - p.n_kv_heads;
      if (gh < p.n_heads) { region = 0; head = gh; }
      else if (gh < p.n_heads + p.n_kv_heads) { region = 1; head = gh - p.n_heads; }
      void* dst;
      size_t off, vt_off = 0;
      if (region == 0) {
        dst = p.q;
        off = ((static_cast<size_t>(b) * p.n_heads + head) * p.R + r) * hd;
      } else {
        dst = region == 1 ? p.k : p.v;
        off = ((static_cast<size_t>(b) * p.n_kv_heads + head) * p.kv_stride + pos) * hd;
        vt_off = (static_cast<size_t>(b) * p.n_kv_heads + head) * hd * p.kv_stride + pos;
      }
      const bool ok = row_ok && nb < p.N;
      // QK-norm: 1 / RMS of this row's head from a first pass over its chunks
      // (the chunks are read again below; the region is uniform across the warp)
      const void* qk_gain = region == 0 ? p.q_gain : (region == 1 ? p.k_gain : nullptr);
      float qk_inv = 1.0f;
      if (qk_gain) {
        float ss = 0.0f;
        for (int c2 = 0; c2 < hd / 32; ++c2) {
          src.load((hh * hd) / 32 + c2, v);
#pragma unroll
          for (int i = 0; i < 32; ++i) ss = fmaf(v[i], v[i], ss);
        }
        qk_inv = rsqrtf(ss / static_cast<float>(hd) + p.qk_eps);
      }
      if (hd == 32) {  // rotate-half pairs (i, i + 16) inside one chunk
        src.load(hh, v);
        if (!ok) continue;
        if (qk_gain) {
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] *= qk_inv * ld_param(qk_gain, p.bias_bf16, i);
        }
        if (p.rope && region < 2) {
          const float2* tab = p.rope_tab + pos;
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const float2 cs = tab[static_cast<size_t>(i) * p.rope_npos];
            const float a = v[i], c2 = v[i + 16];
            v[i] = a * cs.x - c2 * cs.y;
            v[i + 16] = c2 * cs.x + a * cs.y;
          }
        }
        if (region == 2) {
          store_col32(dst, p.out_bf16, vt_off, p.kv_stride, v);
        } else {
          store32(dst, p.out_bf16, off, v, 32);
        }
        continue;
      }
      for (int j2 = 0; j2 < hd / 64; ++j2) {
        float w[32];
        const int ca = (hh * hd) / 32 + j2, cb = ca + hd / 64;
        src.load(ca, v);
        src.load(cb, w);
        if (!ok) continue;
        if (qk_gain) {
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            v[i] *= qk_inv * ld_param(qk_gain, p.bias_bf16, 32 * j2 + i);
            w[i] *= qk_inv * ld_param(qk_gain, p.bias_bf16, hd / 2 + 32 * j2 + i);
          }
        }
        if (p.rope && region < 2) {
          const float2* tab = p.rope_tab + static_cast<size_t>(32 * j2) * p.rope_npos + pos;
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const float2 cs = tab[static_cast<size_t>(i) * p.rope_npos];
            const float a = v[i], c2 = w[i];
            v[i] = a * cs.x - c2 * cs.y;
            w[i] = c2 * cs.x + a * cs.y;
          }
        }
        if (region == 2) {   // V is stored transposed: [b][head][dim][position]
          store_col32(dst, p.out_bf16, vt_off + static_cast<size_t>(32 * j2) * p.kv_stride, p.kv_stride, v);
          store_col32(dst, p.out_bf16, vt_off + static_cast<size_t>(hd / 2 + 32 * j2) * p.kv_stride, p.kv_stride, w);
        } else {
          store32(dst, p.out_bf16, off + 32 * j2, v, 32);
          store32(dst, p.out_bf16, off + hd / 2 + 32 * j2, w, 32);
        }
      }
    }
  } else if constexpr (EPI == EPI_LMHEAD) {
    // sum of exp(l - max) as exp2((l - max) * log2 e)
    constexpr float kLog2e = 1.4426950408889634f;
    float mx = -INFINITY, sum = 0.0f;
    int arg = -1;
    for (int c = c_lo; c < c_hi; ++c) {
      src.load(c, v);
      const int n0 = n_blk * ncols + 32 * c;
      const int nv = min(32, p.N - n0);
      if (!row_ok || nv <= 0) continue;
      if (p.logits) store32(p.logits, 0, static_cast<size_t>(m) * p.ld_logits + n0, v, nv);
      float cmx = -INFINITY;
      int carg = -1;
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        const int n = n0 + i;
        if (i < nv && n != p.mask_id && v[i] > cmx) { cmx = v[i]; carg = n; }
      }
      if (carg < 0) continue;
      const float nm = fmaxf(mx, cmx);
      const float nms = nm * kLog2e;
      float s = (mx == -INFINITY) ? 0.0f : sum * exp2f(fmaf(mx, kLog2e, -nms));
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        const int n = n0 + i;
        if (i < nv && n != p.mask_id) s += exp2f(fmaf(v[i], kLog2e, -nms));
      }
      if (cmx > mx) arg = carg;
      mx = nm;
      sum = s;
    }
    if (row_ok) {
      float* o = p.part + (static_cast<size_t>(m) * p.n_tiles + n_blk * nsplit + part) * 3;
      o[0] = mx;
      o[1] = sum;
      o[2] = __int_as_float(arg);
    }
  } else if constexpr (EPI == EPI_PA_GATE) {
    float s = 0.0f;
    for (int c = 0; c < nch; ++c) {
      src.load(c, v);
      const int n0 = 32 * c;
      const int nv = min(32, p.N - n0);
      if (!row_ok || nv <= 0) continue;
      for (int i = 0; i < nv; ++i) s += silu_f(v[i]) * ld_param(p.vec, p.bias_bf16, n0 + i);
    }
    if (row_ok) static_cast<float*>(p.out)[m] = sigmoid_f(s + ld_param(p.bias, p.bias_bf16, 0));
  }
}

}  // namespace tadm
