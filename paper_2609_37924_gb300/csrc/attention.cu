// Attention over the active rows with a KV context:
//   o = softmax(q k^T / sqrt(hd)) v
// Queries are the rows of the current canvas at absolute positions
// ctx .. ctx+rows-1; keys are positions 0 .. ctx+rows-1 of the layer's K/V
// buffer.  Keys below ctx (committed context) are always visible; the active
// rows see each other bidirectionally, or causally for commit / prefill
// passes.  Query head h reads KV head h / (n_heads / n_kv_heads).
//
// bf16: flash-attention style, one CTA = 64 query rows of one (batch, head),
// 4 warps x 16 rows, key tiles of 64 double-buffered with cp.async,
// QK^T and PV on mma.sync m16n8k16 (fp32 accumulate), online softmax in fp32.
// fp32: one warp per query row on the CUDA cores.
#include "kernels.h"

namespace tadm {
namespace {

constexpr int AM = 64, AN = 64;

__device__ __forceinline__ void cp_async16(void* dst, const void* src, bool pred) {
  const int n = pred ? 16 : 0;
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(dst)), "l"(src), "r"(n) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(smem_u32(p)));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(smem_u32(p)));
}
__device__ __forceinline__ void mma_bf16_16816(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 t = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&t);
}

template <int HD>
__global__ void __launch_bounds__(128) attn_bf16_kernel(const bf16* __restrict__ q, const bf16* __restrict__ k,
                                                        const bf16* __restrict__ v, bf16* __restrict__ o,
                                                        int n_heads, int n_kv_heads, int rows, int ctx,
                                                        int kv_stride, int causal, float scale_log2) {
  constexpr int LD = HD + 8;  // padded smem row (bf16), keeps ldmatrix rows 16-byte aligned
  extern __shared__ __align__(16) uint8_t smem_raw[];
  bf16* sQ = reinterpret_cast<bf16*>(smem_raw);
  bf16* sK = sQ + AM * LD;          // [2][AN][LD]
  bf16* sV = sK + 2 * AN * LD;      // [2][AN][LD]

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int m0 = blockIdx.x * AM, h = blockIdx.y, b = blockIdx.z;
  const int hk = h / (n_heads / n_kv_heads);
  const bf16* qb = q + (static_cast<size_t>(b) * n_heads + h) * rows * HD;
  const bf16* kb = k + (static_cast<size_t>(b) * n_kv_heads + hk) * kv_stride * HD;
  const bf16* vb = v + (static_cast<size_t>(b) * n_kv_heads + hk) * kv_stride * HD;
  const int kv_len = ctx + rows;
  const int kv_end = causal ? min(kv_len, ctx + min(m0 + AM, rows)) : kv_len;
  const int n_tiles = (kv_end + AN - 1) / AN;

  constexpr int CPR = HD / 8;  // 16-byte chunks per row
  for (int i = tid; i < AM * CPR; i += 128) {
    const int r = i / CPR, c = i % CPR;
    const bool ok = m0 + r < rows;
    cp_async16(sQ + r * LD + c * 8, qb + static_cast<size_t>(ok ? m0 + r : 0) * HD + c * 8, ok);
  }
  auto load_kv = [&](int t, int buf) {
    const int n0 = t * AN;
    for (int i = tid; i < AN * CPR; i += 128) {
      const int r = i / CPR, c = i % CPR;
      const bool ok = n0 + r < kv_end;
      const size_t off = static_cast<size_t>(ok ? n0 + r : 0) * HD + c * 8;
      cp_async16(sK + (buf * AN + r) * LD + c * 8, kb + off, ok);
      cp_async16(sV + (buf * AN + r) * LD + c * 8, vb + off, ok);
    }
  };
  if (n_tiles > 0) load_kv(0, 0);
  cp_async_commit();

  float acc[HD / 8][4];
#pragma unroll
  for (int j = 0; j < HD / 8; ++j) acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.0f;
  float mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.0f, 0.0f};
  const int g = lane >> 2, t4 = lane & 3;
  const int qpos0 = ctx + m0 + warp * 16 + g;  // absolute position of this thread's first row
  uint32_t qf[HD / 16][4];

  for (int t = 0; t < n_tiles; ++t) {
    const int buf = t & 1;
    if (t + 1 < n_tiles) load_kv(t + 1, buf ^ 1);
    cp_async_commit();
    cp_async_wait<1>();
    __syncthreads();
    if (t == 0) {
#pragma unroll
      for (int kk = 0; kk < HD / 16; ++kk)
        ldsm_x4(qf[kk], sQ + (warp * 16 + (lane & 15)) * LD + kk * 16 + (lane >> 4) * 8);
    }
    const bf16* Kt = sK + buf * AN * LD;
    const bf16* Vt = sV + buf * AN * LD;
    // S = Q K^T : 16 x 64 per warp
    float s[AN / 8][4];
#pragma unroll
    for (int j = 0; j < AN / 8; ++j) s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.0f;
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
#pragma unroll
      for (int jj = 0; jj < AN / 16; ++jj) {
        uint32_t bfr[4];
        const int key = jj * 16 + (lane & 7) + (lane >> 4) * 8;
        const int dim = kk * 16 + ((lane >> 3) & 1) * 8;
        ldsm_x4(bfr, Kt + key * LD + dim);
        mma_bf16_16816(s[2 * jj], qf[kk], bfr[0], bfr[1]);
        mma_bf16_16816(s[2 * jj + 1], qf[kk], bfr[2], bfr[3]);
      }
    }
    // mask and online softmax (rows g and g+8 of the warp's 16)
    const int n0 = t * AN;
    float tmax[2] = {-INFINITY, -INFINITY};
#pragma unroll
    for (int j = 0; j < AN / 8; ++j) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = n0 + j * 8 + 2 * t4 + (e & 1);
        const int qp = qpos0 + (e >> 1) * 8;
        const bool ok = key < kv_end && (!causal || key < ctx || key <= qp);
        s[j][e] = ok ? s[j][e] * scale_log2 : -INFINITY;
        tmax[e >> 1] = fmaxf(tmax[e >> 1], s[j][e]);
      }
    }
    float corr[2];
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      tmax[r] = fmaxf(tmax[r], __shfl_xor_sync(0xffffffffu, tmax[r], 1));
      tmax[r] = fmaxf(tmax[r], __shfl_xor_sync(0xffffffffu, tmax[r], 2));
      const float mnew = fmaxf(mrow[r], tmax[r]);
      corr[r] = (mnew == -INFINITY) ? 1.0f : exp2f(mrow[r] - mnew);
      mrow[r] = mnew;
      lrow[r] *= corr[r];
    }
    float psum[2] = {0.0f, 0.0f};
#pragma unroll
    for (int j = 0; j < AN / 8; ++j) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float mr = mrow[e >> 1];
        const float p = (mr == -INFINITY) ? 0.0f : exp2f(s[j][e] - mr);
        s[j][e] = p;
        psum[e >> 1] += p;
      }
    }
    lrow[0] += psum[0];
    lrow[1] += psum[1];
#pragma unroll
    for (int j = 0; j < HD / 8; ++j) {
      acc[j][0] *= corr[0]; acc[j][1] *= corr[0];
      acc[j][2] *= corr[1]; acc[j][3] *= corr[1];
    }
    // O += P V
#pragma unroll
    for (int kk = 0; kk < AN / 16; ++kk) {
      uint32_t pa[4];
      pa[0] = pack_bf16(s[2 * kk][0], s[2 * kk][1]);
      pa[1] = pack_bf16(s[2 * kk][2], s[2 * kk][3]);
      pa[2] = pack_bf16(s[2 * kk + 1][0], s[2 * kk + 1][1]);
      pa[3] = pack_bf16(s[2 * kk + 1][2], s[2 * kk + 1][3]);
#pragma unroll
      for (int jj = 0; jj < HD / 16; ++jj) {
        uint32_t vfr[4];
        const int key = kk * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
        const int dim = jj * 16 + (lane >> 4) * 8;
        ldsm_x4_t(vfr, Vt + key * LD + dim);
        mma_bf16_16816(acc[2 * jj], pa, vfr[0], vfr[1]);
        mma_bf16_16816(acc[2 * jj + 1], pa, vfr[2], vfr[3]);
      }
    }
    __syncthreads();
  }
  // finish: row sums across the quad, normalise, store
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 1);
    lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 2);
  }
  const size_t ldo = static_cast<size_t>(n_heads) * HD;
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int row = m0 + warp * 16 + g + r * 8;
    if (row >= rows) continue;
    const float inv = lrow[r] > 0.0f ? 1.0f / lrow[r] : 0.0f;
    bf16* orow = o + (static_cast<size_t>(b) * rows + row) * ldo + static_cast<size_t>(h) * HD;
#pragma unroll
    for (int j = 0; j < HD / 8; ++j) {
      __nv_bfloat162 val = __floats2bfloat162_rn(acc[j][2 * r] * inv, acc[j][2 * r + 1] * inv);
      *reinterpret_cast<__nv_bfloat162*>(orow + j * 8 + 2 * t4) = val;
    }
  }
}

// fp32: one warp per (query row, head, batch); each lane owns hd/32 dims.
template <int HD>
__global__ void __launch_bounds__(128) attn_f32_kernel(const float* __restrict__ q, const float* __restrict__ k,
                                                       const float* __restrict__ v, float* __restrict__ o,
                                                       int n_heads, int n_kv_heads, int rows, int ctx,
                                                       int kv_stride, int causal, float scale) {
  constexpr int PL = HD / 32;
  const int lane = threadIdx.x & 31;
  const int row = blockIdx.x * 4 + (threadIdx.x >> 5);
  const int h = blockIdx.y, b = blockIdx.z;
  if (row >= rows) return;
  const int hk = h / (n_heads / n_kv_heads);
  const float* qr = q + ((static_cast<size_t>(b) * n_heads + h) * rows + row) * HD;
  const float* kb = k + (static_cast<size_t>(b) * n_kv_heads + hk) * kv_stride * HD;
  const float* vb = v + (static_cast<size_t>(b) * n_kv_heads + hk) * kv_stride * HD;
  float qv[PL], acc[PL];
#pragma unroll
  for (int i = 0; i < PL; ++i) { qv[i] = qr[lane + 32 * i]; acc[i] = 0.0f; }
  const int qpos = ctx + row;
  const int kv_end = causal ? qpos + 1 : ctx + rows;
  float m = -INFINITY, l = 0.0f;
  for (int j = 0; j < kv_end; ++j) {
    float d = 0.0f;
#pragma unroll
    for (int i = 0; i < PL; ++i) d += qv[i] * kb[static_cast<size_t>(j) * HD + lane + 32 * i];
    d = warp_sum(d) * scale;
    const float mn = fmaxf(m, d);
    const float c = expf(m - mn), p = expf(d - mn);
    l = l * c + p;
#pragma unroll
    for (int i = 0; i < PL; ++i) acc[i] = acc[i] * c + p * vb[static_cast<size_t>(j) * HD + lane + 32 * i];
    m = mn;
  }
  float* orow = o + (static_cast<size_t>(b) * rows + row) * n_heads * HD + static_cast<size_t>(h) * HD;
#pragma unroll
  for (int i = 0; i < PL; ++i) orow[lane + 32 * i] = acc[i] / l;
}

template <int HD>
cudaError_t launch_bf16(const AttnCall& a, cudaStream_t s) {
  constexpr int LD = HD + 8;
  const size_t smem = static_cast<size_t>(AM + 4 * AN) * LD * sizeof(bf16);
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(attn_bf16_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    attr = true;
  }
  dim3 grid((a.rows + AM - 1) / AM, a.n_heads, a.batch);
  const float scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(HD));
  attn_bf16_kernel<HD><<<grid, 128, smem, s>>>(static_cast<const bf16*>(a.q), static_cast<const bf16*>(a.k),
                                               static_cast<const bf16*>(a.v), static_cast<bf16*>(a.o), a.n_heads,
                                               a.n_kv_heads, a.rows, a.ctx, a.kv_stride, a.causal, scale_log2);
  return cudaGetLastError();
}

template <int HD>
cudaError_t launch_f32(const AttnCall& a, cudaStream_t s) {
  dim3 grid((a.rows + 3) / 4, a.n_heads, a.batch);
  attn_f32_kernel<HD><<<grid, 128, 0, s>>>(static_cast<const float*>(a.q), static_cast<const float*>(a.k),
                                           static_cast<const float*>(a.v), static_cast<float*>(a.o), a.n_heads,
                                           a.n_kv_heads, a.rows, a.ctx, a.kv_stride, a.causal,
                                           1.0f / sqrtf(static_cast<float>(HD)));
  return cudaGetLastError();
}
}  // namespace

const char* attention(const AttnCall& a, cudaStream_t s) {
  if (a.rows <= 0 || a.batch <= 0) return nullptr;
  if (a.n_kv_heads <= 0 || a.n_heads % a.n_kv_heads) return "n_heads must be a multiple of n_kv_heads";
  if (a.kv_stride < a.ctx + a.rows) return "kv_stride smaller than ctx + rows";
  cudaError_t e;
  if (a.bf16) {
    if (a.head_dim == 64) e = launch_bf16<64>(a, s);
    else if (a.head_dim == 128) e = launch_bf16<128>(a, s);
    else return "bf16 attention supports head_dim 64 and 128";
  } else {
    if (a.head_dim == 32) e = launch_f32<32>(a, s);
    else if (a.head_dim == 64) e = launch_f32<64>(a, s);
    else if (a.head_dim == 128) e = launch_f32<128>(a, s);
    else return "fp32 attention supports head_dim 32, 64 and 128";
  }
  return e == cudaSuccess ? nullptr : cudaGetErrorString(e);
}

}  // namespace tadm
