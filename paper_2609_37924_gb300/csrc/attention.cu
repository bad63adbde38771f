// Attention over the active rows with a KV context:
//   o = softmax(q k^T / sqrt(hd)) v
// Queries are the rows of the current canvas at absolute positions
// ctx .. ctx+rows-1; keys are positions 0 .. ctx+rows-1 of the layer's K/V
// buffers.  Keys below ctx (committed context) are always visible; the active
// rows see each other bidirectionally, or causally for commit / prefill
// passes.  The local layers of a Gemma-3 backbone add a sliding window: a
// query at position p sees only keys j with p - j < window (the tcgen05 path
// skips the key tiles below its rows' windows).  Query head h reads KV head
// h / (n_heads / n_kv_heads).
// Layouts: q [B, Hq, rows, hd]; k [B, Hkv, kv_stride, hd];
// v transposed [B, Hkv, hd, kv_stride]; o [B*rows, Hq*hd].
//
// bf16, rows >= 128 (attn_tc_kernel): tcgen05.  One CTA = 128 query rows of
//   one (batch, head).  Warp 0 streams Q once and K / V^T tiles of 128 keys
//   (2-stage ring) with TMA; warp 1 issues S = Q K^T into TMEM and, once the
//   probabilities are in shared memory, O_tile = P V into TMEM; warps 2..5
//   own one query row per thread: masked softmax on the S row, P as bf16
//   into the 128-byte-swizzled operand layout; O accumulates in TMEM across
//   key tiles, rescaled only when a row's running max grows by more than 2^8.
// bf16, short rows (attn_bf16_kernel): mma.sync m16n8k16 flash attention;
//   a CTA takes 64 rows of all query heads of one KV group (one K/V read).
// fp32: one warp per query row on the CUDA cores.
#include <cudaTypedefs.h>
#include <algorithm>
#include <cstdlib>
#include <mutex>

#include "kernels.h"

namespace tadm {
namespace {

// =============================================================== tcgen05 path
constexpr int TQ = 128;      // virtual query rows per CTA (see AttnTcArgs)

// TKV keys per tile: 128, or 64 for hd 128 with few rows, which lets two CTAs
// share an SM.
template <int HD, int TKV>
struct AttnTcCfg {
  static constexpr int Q_BYTES = HD / 64 * 16384;       // HD/64 swizzle atoms of 128 rows x 64
  static constexpr int K_BYTES = HD / 64 * TKV * 128;   // HD/64 atoms of TKV keys x 64
  static constexpr int V_BYTES = TKV / 64 * HD * 128;   // TKV/64 atoms of HD rows x 64 keys
  static constexpr int P_BYTES = TKV / 64 * 16384;      // TKV/64 atoms of 128 rows x 64 keys
  static constexpr int STAGES = 2;
  static constexpr int MIN_BLOCKS = (HD == 64 || TKV == 64) ? 2 : 1;
  // two CTAs per SM leave no room for re-alignment slack: the kernel then
  // requires (and checks) a 1024-byte aligned dynamic base
  static constexpr int SLACK = MIN_BLOCKS == 2 ? 0 : 1024;
  static constexpr int SMEM = SLACK + Q_BYTES + STAGES * (K_BYTES + V_BYTES) + P_BYTES + 256;
  static constexpr int TMEM_COLS = 256;                  // S: [0, TKV), O: [TKV, TKV + HD)
  static_assert(TKV + HD <= TMEM_COLS, "TMEM columns");
};

// Virtual rows: the CTA at blockIdx = (tile + n_vtiles * split, kv head hk,
// batch b) serves virtual rows v = 128 * tile + 0..127, where v = (query head
// within hk's group) * rows + row, so that all query heads of a KV group read
// each K / V tile once, and short canvases fill the 128-row MMA.  With
// `splits` > 1 the keys are cut into splits ranges of tiles_per_split tiles;
// each CTA writes its unnormalised O (fp32), reference max and sum for its
// range to part_o / part_ml, and attn_combine_kernel merges them.
struct AttnTcArgs {
  const bf16* q;
  int rows, ctx, kv_len, n_heads, n_kv_heads, causal;
  int window;        // > 0: keys j < qpos - window + 1 are hidden (sliding window)
  float scale_log2;
  bf16* o;
  int n_vtiles, splits, tiles_per_split;
  float* part_o;     // [splits][B*Hkv][group*rows][HD]
  float2* part_ml;   // [splits][B*Hkv][group*rows]: (reference max in log2 units, sum)
  int* status;
};

// WIN: the sliding window of local layers is in force (a separate
// instantiation, so that the kernel without it carries no window code).
template <int HD, int TKV, bool WIN>
__global__ void __launch_bounds__(192, AttnTcCfg<HD, TKV>::MIN_BLOCKS)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                   const AttnTcArgs args) {
  pdl_enter();
  using C = AttnTcCfg<HD, TKV>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = smem_raw;
  if (C::SLACK) {
    smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  } else if (smem_u32(smem_raw) & 1023) {
    // the swizzled operand layout needs 1024-byte alignment: refuse (uniform exit, nothing started)
    if (threadIdx.x == 0 && args.status) atomicOr(args.status, kErrLayout);
    return;
  }
  uint8_t* sQ = smem;
  uint8_t* sK = sQ + C::Q_BYTES;
  uint8_t* sV = sK + C::STAGES * C::K_BYTES;
  uint8_t* sP = sV + C::STAGES * C::V_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sP + C::P_BYTES);
  uint64_t* q_full = bars;
  uint64_t* kv_full = bars + 1;       // [2]
  uint64_t* kv_empty = bars + 3;      // [2]
  uint64_t* s_full = bars + 5;
  uint64_t* s_free = bars + 6;
  uint64_t* p_full = bars + 7;
  uint64_t* o_full = bars + 8;
  uint64_t* drain = bars + 10;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 11);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int tile = blockIdx.x % args.n_vtiles, split = blockIdx.x / args.n_vtiles;
  const int m0 = tile * TQ, hk = blockIdx.y, b = blockIdx.z;
  const int group = args.n_heads / args.n_kv_heads, n_virt = group * args.rows;
  // causal: the last key any of this CTA's rows may see
  const int v_last = min(m0 + TQ, n_virt) - 1;
  const int r_max = (m0 / args.rows != v_last / args.rows) ? args.rows - 1 : v_last % args.rows;
  const int kv_end = args.causal ? min(args.kv_len, args.ctx + r_max + 1) : args.kv_len;
  // sliding window: no row of this CTA sees a key below the smallest row's window start
  const int r_min = (m0 / args.rows != v_last / args.rows) ? 0 : m0 % args.rows;
  const int kv_begin = WIN ? max(0, args.ctx + r_min - args.window + 1) : 0;
  const int t0 = max(split * args.tiles_per_split, kv_begin / TKV);   // first tile of this CTA
  const int n_tiles = max(0, min((kv_end + TKV - 1) / TKV, (split + 1) * args.tiles_per_split) - t0);

  if (threadIdx.x == 0) {
    mbar_init(q_full, 128);            // the softmax threads stage Q
    for (int s = 0; s < 2; ++s) {
      mbar_init(&kv_full[s], 1);
      mbar_init(&kv_empty[s], 1);
    }
    mbar_init(s_full, 1);
    mbar_init(s_free, 128);
    mbar_init(p_full, 128);
    mbar_init(o_full, 1);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    tma_prefetch_desc(&tmK);
    tma_prefetch_desc(&tmV);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t t_s = tmem, t_o = tmem + TKV;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------------- producer
      int issued0 = 0, issued1 = 0;
      const int z = b * args.n_kv_heads + hk;
      for (int i = 0; i < n_tiles; ++i) {
        const int st = i & 1, j = t0 + i;
        if (!mbar_wait_bounded(&kv_empty[st], ((i >> 1) & 1) ^ 1, abort_flag, args.status)) break;
        mbar_arrive_expect_tx(&kv_full[st], C::K_BYTES + C::V_BYTES);
        for (int s = 0; s < HD / 64; ++s)
          tma_load_3d(sK + st * C::K_BYTES + s * (TKV * 128), &tmK, &kv_full[st], 64 * s, j * TKV, z);
        for (int s = 0; s < TKV / 64; ++s)
          tma_load_3d(sV + st * C::V_BYTES + s * HD * 128, &tmV, &kv_full[st], j * TKV + 64 * s, 0, z);
        if (st) ++issued1; else ++issued0;
        // two stages hold tiles i and i+1; L2 fetches tile i+2 meanwhile
        if (i + 2 < n_tiles) {
          for (int s = 0; s < HD / 64; ++s) tma_prefetch_3d(&tmK, 64 * s, (j + 2) * TKV, z);
          for (int s = 0; s < TKV / 64; ++s) tma_prefetch_3d(&tmV, (j + 2) * TKV + 64 * s, 0, z);
        }
      }
      // every copy started here has landed before the CTA may exit
      volatile int never = 0;
      if (issued0 > 0) mbar_wait_bounded(&kv_full[0], (issued0 - 1) & 1, &never, args.status);
      if (issued1 > 0) mbar_wait_bounded(&kv_full[1], (issued1 - 1) & 1, &never, args.status);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------------------- MMA issuer
      constexpr uint32_t idesc_s = idesc_bf16_f32(TQ, TKV);
      constexpr uint32_t idesc_o = idesc_bf16_f32(TQ, HD);
      bool ok = n_tiles > 0 && mbar_wait_bounded(q_full, 0, abort_flag, args.status);
      const uint32_t q0 = smem_u32(sQ), p0 = smem_u32(sP);
      for (int i = 0; ok && i < n_tiles; ++i) {
        const int st = i & 1;
        if (!mbar_wait_bounded(&kv_full[st], (i >> 1) & 1, abort_flag, args.status)) break;
        if (i > 0 && !mbar_wait_bounded(s_free, (i - 1) & 1, abort_flag, args.status)) break;
        tc_fence_after();
        const uint32_t k0 = smem_u32(sK + st * C::K_BYTES), v0 = smem_u32(sV + st * C::V_BYTES);
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk)
          umma_bf16(t_s, sdesc_kmajor_sw128(q0 + (kk >> 2) * 16384 + (kk & 3) * 32),
                    sdesc_kmajor_sw128(k0 + (kk >> 2) * (TKV * 128) + (kk & 3) * 32), idesc_s, kk != 0);
        umma_commit(s_full);
        // P of tile i is in shared memory and any rescale of O by the softmax
        // threads is complete: O += P V
        if (!mbar_wait_bounded(p_full, i & 1, abort_flag, args.status)) break;
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < TKV / 16; ++kk)
          umma_bf16(t_o, sdesc_kmajor_sw128(p0 + (kk >> 2) * 16384 + (kk & 3) * 32),
                    sdesc_kmajor_sw128(v0 + (kk >> 2) * (HD * 128) + (kk & 3) * 32), idesc_o, (i != 0) || (kk != 0));
        umma_commit(o_full);
        umma_commit(&kv_empty[st]);
      }
      umma_commit(drain);
      volatile int never = 0;
      mbar_wait_bounded(drain, 0, &never, args.status);
    }
  } else {
    // --------------------------------------------------------------- softmax
    // One virtual query row per thread (row = TMEM lane).  O is accumulated
    // in TMEM by the P V MMAs of all key tiles.  The exponentials of every
    // tile use a per-row reference max m_ref (log2 units); m_ref moves only
    // when a tile's max exceeds it by more than 8, and then this thread
    // rescales its row of O (and l) by 2^(m_ref_old - m_ref_new) before the
    // next P V.  Softmax is invariant to the reference, and P <= 2^8 keeps
    // bf16 P and fp32 O exact in range.  The passes use 3-input max and
    // packed fp32-pair arithmetic.
    const int quad = warp & 3;
    const int row = quad * 32 + lane;                 // row within the tile = TMEM lane
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    const int v = m0 + row;
    const bool v_ok = v < n_virt;
    const int qh = hk * group + (v_ok ? v / args.rows : 0);   // query head
    const int qr = v_ok ? v % args.rows : 0;                                         // row of the canvas
    const int qpos = args.ctx + qr;
    // stage this row of Q (zeros past the virtual rows) in the swizzled operand layout
    {
      const uint4* src = reinterpret_cast<const uint4*>(
          args.q + ((static_cast<size_t>(b) * args.n_heads + qh) * args.rows + qr) * HD);
#pragma unroll
      for (int s = 0; s < HD / 64; ++s) {
        uint8_t* dst = sQ + s * 16384 + row * 128;
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          const uint4 val = v_ok ? src[s * 8 + c] : make_uint4(0, 0, 0, 0);
          *reinterpret_cast<uint4*>(dst + ((c ^ (row & 7)) << 4)) = val;
        }
      }
      fence_proxy_async_smem();
      mbar_arrive(q_full);
    }
    float m_ref = -INFINITY, l_run = 0.0f;
    bool ok = true;
    uint8_t* prow0 = sP + row * 128;
    const uint64_t sc2 = f2_pack(args.scale_log2, args.scale_log2);
    for (int i = 0; i < n_tiles; ++i) {
      if (!warp_wait_bounded(s_full, i & 1, abort_flag, args.status)) { ok = false; break; }
      tc_fence_after();
      const int key0 = (t0 + i) * TKV;
      // keys visible to this row: kv_lo <= key < kv_hi (kv_end, or the causal bound; the window start)
      const int kv_hi = args.causal ? min(kv_end, qpos + 1) : kv_end;
      const int lim = kv_hi - key0;                                   // visible keys of this tile: [lo, lim)
      const int lo = WIN ? qpos - args.window + 1 - key0 : 0;
      const bool masked = __any_sync(0xffffffffu, lim < TKV || (WIN && lo > 0));   // warp-uniform path choice
      // pass 1: row max over the tile, 64 columns per TMEM round trip
      float mxa[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};   // independent chains
#pragma unroll
      for (int c = 0; c < TKV / 64; ++c) {
        uint32_t ra[32], rb[32];
        tmem_ld32_nowait(t_s + lane_off + 64 * c, ra);
        tmem_ld32_nowait(t_s + lane_off + 64 * c + 32, rb);
        tmem_wait_ld(ra);
        tmem_bind(rb);
        if (masked) {
#pragma unroll
          for (int k = 0; k < 32; ++k)
            mxa[k & 3] = fmax3(mxa[k & 3],
                               64 * c + k < lim && 64 * c + k >= lo ? __uint_as_float(ra[k]) : -INFINITY,
                               64 * c + 32 + k < lim && 64 * c + 32 + k >= lo ? __uint_as_float(rb[k]) : -INFINITY);
        } else {
#pragma unroll
          for (int k = 0; k < 32; ++k) mxa[k & 3] = fmax3(mxa[k & 3], __uint_as_float(ra[k]), __uint_as_float(rb[k]));
        }
      }
      const float m_tile = fmax3(fmaxf(mxa[0], mxa[1]), mxa[2], mxa[3]) * args.scale_log2;
      float m_new = m_ref, factor = 1.0f;
      if (m_ref == -INFINITY) {
        m_new = m_tile;                          // every earlier exponential was 0: nothing to rescale
      } else if (m_tile > m_ref + 8.0f) {
        m_new = m_tile;
        factor = ex2_approx(m_ref - m_tile);     // < 2^-8
      }
      if (__any_sync(0xffffffffu, factor != 1.0f)) {
        // O holds tiles 0 .. i-1 once the P V of tile i-1 is done (i >= 1 here)
        if (!warp_wait_bounded(o_full, (i - 1) & 1, abort_flag, args.status)) { ok = false; break; }
        tc_fence_after();
#pragma unroll
        for (int c = 0; c < HD / 32; ++c) {
          uint32_t ra[32];
          tmem_ld32_nowait(t_o + lane_off + 32 * c, ra);
          tmem_wait_ld(ra);
#pragma unroll
          for (int k = 0; k < 32; ++k) ra[k] = __float_as_uint(__uint_as_float(ra[k]) * factor);
          tmem_st32(t_o + lane_off + 32 * c, ra);
        }
        tmem_wait_st();
        l_run *= factor;
      }
      // pass 2: P = 2^(s * scale - m_new) as bf16 into the swizzled A-operand layout, 32 columns per trip
      const uint64_t negm2 = f2_pack(-m_new, -m_new);
      uint64_t ps2[2] = {0, 0};                  // packed partial sums, two chains
#pragma unroll
      for (int c = 0; c < TKV / 32; ++c) {
        uint32_t ra[32];
        tmem_ld32_nowait(t_s + lane_off + 32 * c, ra);
        tmem_wait_ld(ra);
        uint32_t pk[16];
#pragma unroll
        for (int k = 0; k < 32; k += 2) {
          float x0, x1;
          f2_unpack(f2_fma(f2_pack(__uint_as_float(ra[k]), __uint_as_float(ra[k + 1])), sc2, negm2), x0, x1);
          float p0 = ex2_approx(x0), p1 = ex2_approx(x1);
          if (masked) {
            p0 = 32 * c + k < lim && 32 * c + k >= lo ? p0 : 0.0f;
            p1 = 32 * c + k + 1 < lim && 32 * c + k + 1 >= lo ? p1 : 0.0f;
          }
          ps2[(k >> 1) & 1] = f2_add(ps2[(k >> 1) & 1], f2_pack(p0, p1));
          __nv_bfloat162 t = __floats2bfloat162_rn(p0, p1);
          pk[k / 2] = *reinterpret_cast<uint32_t*>(&t);
        }
        // keys 32c .. 32c+31: atom (32c / 64), 16-byte chunks (32c % 64) / 8 .. +3
        uint8_t* atom = prow0 + (c >> 1) * 16384;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int chunk = (c & 1) * 4 + q;
          *reinterpret_cast<uint4*>(atom + ((chunk ^ (row & 7)) << 4)) =
              make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
        }
      }
      float a0, a1, b0, b1;
      f2_unpack(ps2[0], a0, a1);
      f2_unpack(ps2[1], b0, b1);
      l_run += (a0 + a1) + (b0 + b1);
      m_ref = m_new;
      tc_fence_before();
      fence_proxy_async_smem();
      mbar_arrive(s_free);
      mbar_arrive(p_full);
    }
    const size_t bk = static_cast<size_t>(b) * args.n_kv_heads + hk;
    if (args.splits > 1 && ok && n_tiles == 0) {
      // no key of this split: an empty partial
      if (v_ok) {
        const size_t pr = (static_cast<size_t>(split) * args.n_kv_heads * gridDim.z + bk) * n_virt + v;
        float4* po = reinterpret_cast<float4*>(args.part_o + pr * HD);
        for (int k = 0; k < HD / 4; ++k) po[k] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
        args.part_ml[pr] = make_float2(-INFINITY, 0.0f);
      }
    } else if (ok && n_tiles > 0 && warp_wait_bounded(o_full, (n_tiles - 1) & 1, abort_flag, args.status)) {
      tc_fence_after();
      if (args.splits > 1) {
        const size_t pr = (static_cast<size_t>(split) * args.n_kv_heads * gridDim.z + bk) * n_virt + v;
        float4* po = reinterpret_cast<float4*>(args.part_o + pr * HD);
#pragma unroll
        for (int c = 0; c < HD / 32; ++c) {
          uint32_t ra[32];
          tmem_ld32_nowait(t_o + lane_off + 32 * c, ra);
          tmem_wait_ld(ra);
          if (v_ok) {
#pragma unroll
            for (int k = 0; k < 32; k += 4)
              po[(32 * c + k) / 4] = make_float4(__uint_as_float(ra[k]), __uint_as_float(ra[k + 1]),
                                                 __uint_as_float(ra[k + 2]), __uint_as_float(ra[k + 3]));
          }
        }
        if (v_ok) args.part_ml[pr] = make_float2(m_ref, l_run);
      } else {
        const float inv = l_run > 0.0f ? 1.0f / l_run : 0.0f;
        bf16* orow = args.o + (static_cast<size_t>(b) * args.rows + qr) * args.n_heads * HD + static_cast<size_t>(qh) * HD;
#pragma unroll
        for (int c = 0; c < HD / 32; ++c) {
          uint32_t ra[32];
          tmem_ld32_nowait(t_o + lane_off + 32 * c, ra);
          tmem_wait_ld(ra);
          if (v_ok) {
#pragma unroll
            for (int k = 0; k < 32; k += 8) {
              __nv_bfloat162 w0 = __floats2bfloat162_rn(__uint_as_float(ra[k]) * inv, __uint_as_float(ra[k + 1]) * inv);
              __nv_bfloat162 w1 = __floats2bfloat162_rn(__uint_as_float(ra[k + 2]) * inv, __uint_as_float(ra[k + 3]) * inv);
              __nv_bfloat162 w2 = __floats2bfloat162_rn(__uint_as_float(ra[k + 4]) * inv, __uint_as_float(ra[k + 5]) * inv);
              __nv_bfloat162 w3 = __floats2bfloat162_rn(__uint_as_float(ra[k + 6]) * inv, __uint_as_float(ra[k + 7]) * inv);
              *reinterpret_cast<uint4*>(orow + 32 * c + k) =
                  make_uint4(*reinterpret_cast<uint32_t*>(&w0), *reinterpret_cast<uint32_t*>(&w1),
                             *reinterpret_cast<uint32_t*>(&w2), *reinterpret_cast<uint32_t*>(&w3));
            }
          }
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

// ------------------------------------------------------------ pipelined variant
// The same computation without key splits or a window, with the tensor pipe
// and the softmax overlapped: 64-key tiles, S double-buffered in TMEM (S0,
// S1, then O: 2 * 64 + hd of the 256 columns; two CTAs per SM for hd 64, one
// for hd 128, whose four stages of 32 KB fill the shared memory) and P
// double-buffered in shared memory, four K / V stages.  The MMA thread
// issues S(i) as soon as the softmax has released its S buffer (tile i - 2),
// then O += P(i-1) V(i-1): while the softmax threads exponentiate tile i,
// the tensor pipe already computes S(i+1).  Ordering facts the softmax relies
// on (tcgen05 operations of one thread complete in issue order): P V(i-2) is
// issued before S(i), so when S(i) is complete the P buffer of tile i and
// the O accumulator up to tile i-2 are settled; a rescale of O at tile i
// waits for P V(i-1) on o_full.
template <int HD_>
struct AttnDbCfg {
  static constexpr int HD = HD_, TKV = 64, STAGES = 4;
  static constexpr int MIN_BLOCKS = HD == 64 ? 2 : 1;
  static constexpr int Q_BYTES = HD / 64 * 16384;     // HD/64 swizzle atoms of 128 rows x 64 dims
  static constexpr int K_BYTES = HD / 64 * TKV * 128; // HD/64 atoms of 64 keys x 64 dims
  static constexpr int V_BYTES = HD * 128;            // HD dims x 64 keys (V^T)
  static constexpr int P_BYTES = 16384;               // 128 rows x 64 keys
  static constexpr int SMEM = Q_BYTES + STAGES * (K_BYTES + V_BYTES) + 2 * P_BYTES + 256;
  static constexpr int TMEM_COLS = 256;               // S0 [0, 64), S1 [64, 128), O [128, 128 + HD)
  static_assert(2 * TKV + HD <= TMEM_COLS, "TMEM columns");
};

template <int HD_>
__global__ void __launch_bounds__(192, AttnDbCfg<HD_>::MIN_BLOCKS)
    attn_db_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                   const AttnTcArgs args) {
  pdl_enter();
  using C = AttnDbCfg<HD_>;
  constexpr int HD = C::HD, TKV = C::TKV, NST = C::STAGES;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = smem_raw;
  if (smem_u32(smem_raw) & 1023) {
    // the swizzled operand layout needs 1024-byte alignment: refuse (uniform exit, nothing started)
    if (threadIdx.x == 0 && args.status) atomicOr(args.status, kErrLayout);
    return;
  }
  uint8_t* sQ = smem;
  uint8_t* sK = sQ + C::Q_BYTES;
  uint8_t* sV = sK + NST * C::K_BYTES;
  uint8_t* sP = sV + NST * C::V_BYTES;                 // two P buffers
  uint64_t* bars = reinterpret_cast<uint64_t*>(sP + 2 * C::P_BYTES);
  uint64_t* q_full = bars;
  uint64_t* kv_full = bars + 1;        // [NST]
  uint64_t* kv_empty = bars + 5;       // [NST]
  uint64_t* s_full = bars + 9;         // [2]
  uint64_t* s_free = bars + 11;        // [2]
  uint64_t* p_full = bars + 13;        // [2]
  uint64_t* o_full = bars + 15;        // one completion per P V
  uint64_t* drain = bars + 16;
  uint64_t* o_done = bars + 17;        // the last P V is complete
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 18);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int m0 = blockIdx.x * TQ, hk = blockIdx.y, b = blockIdx.z;
  const int group = args.n_heads / args.n_kv_heads, n_virt = group * args.rows;
  const int v_last = min(m0 + TQ, n_virt) - 1;
  const int r_max = (m0 / args.rows != v_last / args.rows) ? args.rows - 1 : v_last % args.rows;
  const int kv_end = args.causal ? min(args.kv_len, args.ctx + r_max + 1) : args.kv_len;
  const int n_tiles = (kv_end + TKV - 1) / TKV;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 128);
    for (int s = 0; s < NST; ++s) {
      mbar_init(&kv_full[s], 1);
      mbar_init(&kv_empty[s], 1);
    }
    for (int s = 0; s < 2; ++s) {
      mbar_init(&s_full[s], 1);
      mbar_init(&s_free[s], 128);
      mbar_init(&p_full[s], 128);
    }
    mbar_init(o_full, 1);
    mbar_init(drain, 1);
    mbar_init(o_done, 1);
    *abort_flag = 0;
    fence_mbar_init();
    tma_prefetch_desc(&tmK);
    tma_prefetch_desc(&tmV);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t t_o = tmem + 2 * TKV;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------------------- producer
      int issued[NST];
      for (int s = 0; s < NST; ++s) issued[s] = 0;
      const int z = b * args.n_kv_heads + hk;
      for (int i = 0; i < n_tiles; ++i) {
        const int st = i % NST;
        if (!mbar_wait_bounded(&kv_empty[st], ((i / NST) & 1) ^ 1, abort_flag, args.status)) break;
        mbar_arrive_expect_tx(&kv_full[st], C::K_BYTES + C::V_BYTES);
        for (int s = 0; s < HD / 64; ++s)
          tma_load_3d(sK + st * C::K_BYTES + s * (TKV * 128), &tmK, &kv_full[st], 64 * s, i * TKV, z);
        tma_load_3d(sV + st * C::V_BYTES, &tmV, &kv_full[st], i * TKV, 0, z);
        ++issued[st];
        if (i + NST < n_tiles) {     // the stage ring holds tiles i .. i+3; L2 fetches tile i+4 meanwhile
          for (int s = 0; s < HD / 64; ++s) tma_prefetch_3d(&tmK, 64 * s, (i + NST) * TKV, z);
          tma_prefetch_3d(&tmV, (i + NST) * TKV, 0, z);
        }
      }
      // every copy started here has landed before the CTA may exit
      volatile int never = 0;
      for (int s = 0; s < NST; ++s)
        if (issued[s] > 0) mbar_wait_bounded(&kv_full[s], (issued[s] - 1) & 1, &never, args.status);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------------------- MMA issuer
      constexpr uint32_t idesc_s = idesc_bf16_f32(TQ, TKV);
      constexpr uint32_t idesc_o = idesc_bf16_f32(TQ, HD);
      bool ok = n_tiles > 0 && mbar_wait_bounded(q_full, 0, abort_flag, args.status);
      const uint32_t q0 = smem_u32(sQ);
      for (int i = 0; ok && i <= n_tiles; ++i) {
        if (i < n_tiles) {
          // S(i) = Q K(i)^T into S buffer i & 1, once the softmax has released it (tile i - 2)
          const int st = i % NST, sb = i & 1;
          if (!mbar_wait_bounded(&kv_full[st], (i / NST) & 1, abort_flag, args.status)) break;
          if (i >= 2 && !mbar_wait_bounded(&s_free[sb], ((i - 2) >> 1) & 1, abort_flag, args.status)) break;
          tc_fence_after();
          const uint32_t k0 = smem_u32(sK + st * C::K_BYTES);
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk)
            umma_bf16(tmem + sb * TKV, sdesc_kmajor_sw128(q0 + (kk >> 2) * 16384 + (kk & 3) * 32),
                      sdesc_kmajor_sw128(k0 + (kk >> 2) * (TKV * 128) + (kk & 3) * 32), idesc_s, kk != 0);
          umma_commit(&s_full[sb]);
        }
        if (i >= 1) {
          // O += P(j) V(j) for the previous tile, once its probabilities are in shared memory
          const int j = i - 1, pb = j & 1, st = j % NST;
          if (!mbar_wait_bounded(&p_full[pb], (j >> 1) & 1, abort_flag, args.status)) break;
          tc_fence_after();
          const uint32_t p0 = smem_u32(sP + pb * C::P_BYTES), v0 = smem_u32(sV + st * C::V_BYTES);
#pragma unroll
          for (int kk = 0; kk < TKV / 16; ++kk)
            umma_bf16(t_o, sdesc_kmajor_sw128(p0 + kk * 32), sdesc_kmajor_sw128(v0 + kk * 32), idesc_o,
                      (j != 0) || (kk != 0));
          umma_commit(o_full);
          umma_commit(&kv_empty[st]);
          if (j == n_tiles - 1) umma_commit(o_done);
        }
      }
      umma_commit(drain);
      volatile int never = 0;
      mbar_wait_bounded(drain, 0, &never, args.status);
    }
  } else {
    // --------------------------------------------------------------- softmax
    // One virtual query row per thread (row = TMEM lane), the reference-max
    // scheme of attn_tc_kernel (O rescaled only when a tile's max exceeds the
    // reference by more than 8 in log2 units).
    const int quad = warp & 3;
    const int row = quad * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    const int v = m0 + row;
    const bool v_ok = v < n_virt;
    const int qh = hk * group + (v_ok ? v / args.rows : 0);
    const int qr = v_ok ? v % args.rows : 0;
    const int qpos = args.ctx + qr;
    {
      const uint4* src = reinterpret_cast<const uint4*>(
          args.q + ((static_cast<size_t>(b) * args.n_heads + qh) * args.rows + qr) * HD);
#pragma unroll
      for (int s = 0; s < HD / 64; ++s) {
        uint8_t* dst = sQ + s * 16384 + row * 128;
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          const uint4 val = v_ok ? src[s * 8 + c] : make_uint4(0, 0, 0, 0);
          *reinterpret_cast<uint4*>(dst + ((c ^ (row & 7)) << 4)) = val;
        }
      }
      fence_proxy_async_smem();
      mbar_arrive(q_full);
    }
    float m_ref = -INFINITY, l_run = 0.0f;
    bool ok = true;
    const uint64_t sc2 = f2_pack(args.scale_log2, args.scale_log2);
    const int kv_hi = args.causal ? min(kv_end, qpos + 1) : kv_end;
    for (int i = 0; i < n_tiles; ++i) {
      const int sb = i & 1;
      if (!warp_wait_bounded(&s_full[sb], (i >> 1) & 1, abort_flag, args.status)) { ok = false; break; }
      tc_fence_after();
      const uint32_t t_s = tmem + sb * TKV + lane_off;
      const int lim = kv_hi - i * TKV;                                // visible keys of this tile
      const bool masked = __any_sync(0xffffffffu, lim < TKV);
      uint32_t ra[32], rb[32];
      tmem_ld32_nowait(t_s, ra);
      tmem_ld32_nowait(t_s + 32, rb);
      tmem_wait_ld(ra);
      tmem_bind(rb);
      // S is in registers: its TMEM buffer goes back to the MMA thread (S(i+2)) at once
      tc_fence_before();
      mbar_arrive(&s_free[sb]);
      // pass 1: row max over the tile (both halves stay in registers for pass 2)
      float mxa[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
      if (masked) {
#pragma unroll
        for (int k = 0; k < 32; ++k)
          mxa[k & 3] = fmax3(mxa[k & 3], k < lim ? __uint_as_float(ra[k]) : -INFINITY,
                             32 + k < lim ? __uint_as_float(rb[k]) : -INFINITY);
      } else {
#pragma unroll
        for (int k = 0; k < 32; ++k) mxa[k & 3] = fmax3(mxa[k & 3], __uint_as_float(ra[k]), __uint_as_float(rb[k]));
      }
      const float m_tile = fmax3(fmaxf(mxa[0], mxa[1]), mxa[2], mxa[3]) * args.scale_log2;
      float m_new = m_ref, factor = 1.0f;
      if (m_ref == -INFINITY) {
        m_new = m_tile;
      } else if (m_tile > m_ref + 8.0f) {
        m_new = m_tile;
        factor = ex2_approx(m_ref - m_tile);
      }
      if (__any_sync(0xffffffffu, factor != 1.0f)) {
        // O holds tiles 0 .. i-1 once P V(i-1) is complete (i >= 1 here)
        if (!warp_wait_bounded(o_full, (i - 1) & 1, abort_flag, args.status)) { ok = false; break; }
        tc_fence_after();
#pragma unroll
        for (int c = 0; c < HD / 32; ++c) {
          uint32_t ro[32];
          tmem_ld32_nowait(t_o + lane_off + 32 * c, ro);
          tmem_wait_ld(ro);
#pragma unroll
          for (int k = 0; k < 32; ++k) ro[k] = __float_as_uint(__uint_as_float(ro[k]) * factor);
          tmem_st32(t_o + lane_off + 32 * c, ro);
        }
        tmem_wait_st();
        l_run *= factor;
      }
      // pass 2: P = 2^(s * scale - m_new) as bf16 into P buffer i & 1 (free: P V(i-2) is complete)
      uint8_t* prow = sP + sb * C::P_BYTES + row * 128;
      const uint64_t negm2 = f2_pack(-m_new, -m_new);
      uint64_t ps2[2] = {0, 0};
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        const uint32_t* r = c ? rb : ra;
        uint32_t pk[16];
#pragma unroll
        for (int k = 0; k < 32; k += 2) {
          float x0, x1;
          f2_unpack(f2_fma(f2_pack(__uint_as_float(r[k]), __uint_as_float(r[k + 1])), sc2, negm2), x0, x1);
          float p0 = ex2_approx(x0), p1 = ex2_approx(x1);
          if (masked) {
            p0 = 32 * c + k < lim ? p0 : 0.0f;
            p1 = 32 * c + k + 1 < lim ? p1 : 0.0f;
          }
          ps2[(k >> 1) & 1] = f2_add(ps2[(k >> 1) & 1], f2_pack(p0, p1));
          __nv_bfloat162 t = __floats2bfloat162_rn(p0, p1);
          pk[k / 2] = *reinterpret_cast<uint32_t*>(&t);
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int chunk = c * 4 + q;
          *reinterpret_cast<uint4*>(prow + ((chunk ^ (row & 7)) << 4)) =
              make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
        }
      }
      float a0, a1, b0, b1;
      f2_unpack(ps2[0], a0, a1);
      f2_unpack(ps2[1], b0, b1);
      l_run += (a0 + a1) + (b0 + b1);
      m_ref = m_new;
      fence_proxy_async_smem();
      mbar_arrive(&p_full[sb]);
    }
    // o_done, not o_full: at this point P V(n-2) may still be running as well
    if (ok && n_tiles > 0 && warp_wait_bounded(o_done, 0, abort_flag, args.status)) {
      tc_fence_after();
      const float inv = l_run > 0.0f ? 1.0f / l_run : 0.0f;
      bf16* orow = args.o + (static_cast<size_t>(b) * args.rows + qr) * args.n_heads * HD + static_cast<size_t>(qh) * HD;
#pragma unroll
      for (int c = 0; c < HD / 32; ++c) {
        uint32_t ro[32];
        tmem_ld32_nowait(t_o + lane_off + 32 * c, ro);
        tmem_wait_ld(ro);
        if (v_ok) {
#pragma unroll
          for (int k = 0; k < 32; k += 8) {
            __nv_bfloat162 w0 = __floats2bfloat162_rn(__uint_as_float(ro[k]) * inv, __uint_as_float(ro[k + 1]) * inv);
            __nv_bfloat162 w1 = __floats2bfloat162_rn(__uint_as_float(ro[k + 2]) * inv, __uint_as_float(ro[k + 3]) * inv);
            __nv_bfloat162 w2 = __floats2bfloat162_rn(__uint_as_float(ro[k + 4]) * inv, __uint_as_float(ro[k + 5]) * inv);
            __nv_bfloat162 w3 = __floats2bfloat162_rn(__uint_as_float(ro[k + 6]) * inv, __uint_as_float(ro[k + 7]) * inv);
            *reinterpret_cast<uint4*>(orow + 32 * c + k) =
                make_uint4(*reinterpret_cast<uint32_t*>(&w0), *reinterpret_cast<uint32_t*>(&w1),
                           *reinterpret_cast<uint32_t*>(&w2), *reinterpret_cast<uint32_t*>(&w3));
          }
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

// Merges the split partials of one virtual row per warp, in split order:
// m* = max m_s, O = sum 2^(m_s - m*) O_s / sum 2^(m_s - m*) l_s.
template <int HD>
__global__ void __launch_bounds__(256) attn_combine_kernel(const float* __restrict__ part_o,
                                                           const float2* __restrict__ part_ml, int splits,
                                                           int n_bk, int n_virt, int rows, int n_heads,
                                                           int n_kv_heads, bf16* __restrict__ o) {
  pdl_enter();
  constexpr int PL = HD / 32;   // dims per lane
  const int lane = threadIdx.x & 31;
  const int g = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (g >= n_bk * n_virt) return;
  const size_t stride = static_cast<size_t>(n_bk) * n_virt;
  float mx = -INFINITY;
  for (int s = 0; s < splits; ++s) mx = fmaxf(mx, part_ml[s * stride + g].x);
  float acc[PL];
#pragma unroll
  for (int k = 0; k < PL; ++k) acc[k] = 0.0f;
  float L = 0.0f;
  if (mx != -INFINITY) {
    for (int s = 0; s < splits; ++s) {
      const float2 ml = part_ml[s * stride + g];
      const float w = ml.x == -INFINITY ? 0.0f : ex2_approx(ml.x - mx);
      L = fmaf(w, ml.y, L);
      const float* src = part_o + (s * stride + g) * HD + lane * PL;
#pragma unroll
      for (int k = 0; k < PL; ++k) acc[k] = fmaf(w, src[k], acc[k]);
    }
  }
  const float inv = L > 0.0f ? 1.0f / L : 0.0f;
  const int bk = g / n_virt, v = g - bk * n_virt;
  const int group = n_heads / n_kv_heads;
  const int b = bk / n_kv_heads, hk = bk - b * n_kv_heads;
  const int h = hk * group + v / rows, r = v % rows;
  bf16* orow = o + (static_cast<size_t>(b) * rows + r) * n_heads * HD + static_cast<size_t>(h) * HD + lane * PL;
#pragma unroll
  for (int k = 0; k < PL; k += 2)
    *reinterpret_cast<__nv_bfloat162*>(orow + k) = __floats2bfloat162_rn(acc[k] * inv, acc[k + 1] * inv);
}

PFN_cuTensorMapEncodeTiled_v12000 g_enc = nullptr;
std::once_flag g_enc_once;

bool encoder() {
  std::call_once(g_enc_once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_enc = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  });
  return g_enc != nullptr;
}

// 3-D bf16 map: dims {d0 (contiguous), d1, d2}, byte strides {s1, s2}, box {64, box1, 1}, 128-byte swizzle.
bool map3d(CUtensorMap* m, const void* ptr, uint64_t d0, uint64_t d1, uint64_t d2, uint64_t s1, uint64_t s2,
           uint32_t box1) {
  cuuint64_t dims[3] = {d0, d1, d2};
  cuuint64_t strides[2] = {s1, s2};
  cuuint32_t box[3] = {64, box1, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return g_enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(ptr), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int HD, int TKV, bool WIN>
const char* launch_tc_win(const AttnCall& a, cudaStream_t s) {
  using C = AttnTcCfg<HD, TKV>;
  if (!encoder()) return "cuTensorMapEncodeTiled is unavailable";
  const int kv_len = a.ctx + a.rows;
  CUtensorMap mk, mv;
  // K: {hd, kv_len, B*Hkv}; V^T: {kv_len, hd, B*Hkv} -- positions past kv_len read zeros
  if (!map3d(&mk, a.k, HD, kv_len, static_cast<uint64_t>(a.batch) * a.n_kv_heads, HD * 2ull,
             static_cast<uint64_t>(a.kv_stride) * HD * 2, TKV) ||
      !map3d(&mv, a.v, kv_len, HD, static_cast<uint64_t>(a.batch) * a.n_kv_heads, a.kv_stride * 2ull,
             static_cast<uint64_t>(a.kv_stride) * HD * 2, HD))
    return "attention tensor map encode failed";
  static int n_sms = 0;
  if (n_sms == 0) {
    if (cudaFuncSetAttribute(attn_tc_kernel<HD, TKV, WIN>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM) !=
        cudaSuccess)
      return "attention smem attribute failed";
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n_sms, cudaDevAttrMultiProcessorCount, dev);
    if (n_sms <= 0) n_sms = 1;
  }
  const int group = a.n_heads / a.n_kv_heads, n_virt = group * a.rows;
  const int n_vtiles = (n_virt + TQ - 1) / TQ;
  const int base = n_vtiles * a.n_kv_heads * a.batch;
  const int kv_tiles = (kv_len + TKV - 1) / TKV;
  // split the keys only into as many ranges as the resident CTA slots leave
  // room for (splitting adds partial traffic and a merge, it only pays for
  // idle SMs): every split keeps >= 3 tiles and its fp32 partials fit the
  // caller's scratch
  int splits = 1;
  // a window leaves each CTA only its window's tiles: no key splits then
  if (a.part && a.part_bytes > 0 && !WIN) {
    const int slots = C::MIN_BLOCKS * n_sms;
    const size_t per_split = static_cast<size_t>(a.batch) * a.n_kv_heads * n_virt * (HD + 2) * sizeof(float);
    splits = std::min(std::min(slots / base, kv_tiles / 3), 8);
    while (splits > 1 && static_cast<size_t>(splits) * per_split > a.part_bytes) --splits;
    if (splits < 1) splits = 1;
  }
  const int tps = (kv_tiles + splits - 1) / splits;
  splits = (kv_tiles + tps - 1) / tps;
  float* part_o = static_cast<float*>(a.part);
  float2* part_ml = reinterpret_cast<float2*>(part_o + static_cast<size_t>(splits) * a.batch * a.n_kv_heads * n_virt * HD);
  AttnTcArgs args{static_cast<const bf16*>(a.q), a.rows, a.ctx, kv_len, a.n_heads, a.n_kv_heads, a.causal, a.window,
                  1.4426950408889634f / sqrtf(static_cast<float>(HD)), static_cast<bf16*>(a.o),
                  n_vtiles, splits, tps, part_o, part_ml, a.status};
  dim3 grid(n_vtiles * splits, a.n_kv_heads, a.batch);
  launch_pdl(attn_tc_kernel<HD, TKV, WIN>, grid, 192, C::SMEM, s, mk, mv, args);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cudaGetErrorString(e);
  if (splits > 1) {
    const int n_bk = a.batch * a.n_kv_heads;
    const int rows_total = n_bk * n_virt;
    launch_pdl(attn_combine_kernel<HD>, (rows_total + 7) / 8, 256, 0, s, part_o, part_ml, splits, n_bk, n_virt, a.rows,
                                                               a.n_heads, a.n_kv_heads, static_cast<bf16*>(a.o));
    e = cudaGetLastError();
    if (e != cudaSuccess) return cudaGetErrorString(e);
  }
  return nullptr;
}

// The pipelined hd-64 kernel: whenever no key split is wanted (the CTAs of
// the launch fill the SMs) and no window hides keys.  TADM_ATTN_DB=0 keeps
// attn_tc_kernel for every shape.
bool attn_db_enabled() {
  static const bool on = [] {
    const char* e = getenv("TADM_ATTN_DB");
    return !(e && e[0] == '0');
  }();
  return on;
}

template <int HD>
const char* launch_db(const AttnCall& a, cudaStream_t s) {
  using C = AttnDbCfg<HD>;
  if (!encoder()) return "cuTensorMapEncodeTiled is unavailable";
  const int kv_len = a.ctx + a.rows;
  CUtensorMap mk, mv;
  if (!map3d(&mk, a.k, C::HD, kv_len, static_cast<uint64_t>(a.batch) * a.n_kv_heads, C::HD * 2ull,
             static_cast<uint64_t>(a.kv_stride) * C::HD * 2, C::TKV) ||
      !map3d(&mv, a.v, kv_len, C::HD, static_cast<uint64_t>(a.batch) * a.n_kv_heads, a.kv_stride * 2ull,
             static_cast<uint64_t>(a.kv_stride) * C::HD * 2, C::HD))
    return "attention tensor map encode failed";
  static bool attr = false;
  if (!attr) {
    if (cudaFuncSetAttribute(attn_db_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM) != cudaSuccess)
      return "attention smem attribute failed";
    attr = true;
  }
  const int group = a.n_heads / a.n_kv_heads, n_virt = group * a.rows;
  const int n_vtiles = (n_virt + TQ - 1) / TQ;
  AttnTcArgs args{static_cast<const bf16*>(a.q), a.rows, a.ctx, kv_len, a.n_heads, a.n_kv_heads, a.causal, 0,
                  1.4426950408889634f / sqrtf(static_cast<float>(C::HD)), static_cast<bf16*>(a.o),
                  n_vtiles, 1, 0, nullptr, nullptr, a.status};
  launch_pdl(attn_db_kernel<HD>, dim3(n_vtiles, a.n_kv_heads, a.batch), 192, C::SMEM, s, mk, mv, args);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? nullptr : cudaGetErrorString(e);
}

// the windowed kernel only where the window hides keys (window < ctx + rows)
template <int HD, int TKV>
const char* launch_tc(const AttnCall& a, cudaStream_t s) {
  return a.window > 0 && a.window < a.ctx + a.rows ? launch_tc_win<HD, TKV, true>(a, s)
                                                   : launch_tc_win<HD, TKV, false>(a, s);
}

// ============================================================= mma.sync path
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
                                                        const bf16* __restrict__ vt, bf16* __restrict__ o,
                                                        int n_heads, int n_kv_heads, int rows, int ctx,
                                                        int kv_stride, int causal, int window, float scale_log2) {
  pdl_enter();
  constexpr int LD = HD + 8;   // padded smem row of Q / K (bf16)
  constexpr int LDV = AN + 8;  // padded smem row of V^T (one head dim, AN keys)
  extern __shared__ __align__(16) uint8_t smem_raw[];
  bf16* sQ = reinterpret_cast<bf16*>(smem_raw);
  bf16* sK = sQ + AM * LD;          // [2][AN][LD]
  bf16* sV = sK + 2 * AN * LD;      // [2][HD][LDV]

  // One CTA serves AM "virtual rows" v = (query head within the KV group) *
  // rows + row of one (batch, KV head): the group's query heads share every
  // K / V tile, which is read once for all of them.
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int m0 = blockIdx.x * AM, hk = blockIdx.y, b = blockIdx.z;
  const int group = n_heads / n_kv_heads, n_virt = group * rows;
  const bf16* kb = k + (static_cast<size_t>(b) * n_kv_heads + hk) * kv_stride * HD;
  const bf16* vb = vt + (static_cast<size_t>(b) * n_kv_heads + hk) * HD * kv_stride;
  const int kv_len = ctx + rows;
  // causal: the last key any of this CTA's rows may see
  const int v_last = min(m0 + AM, n_virt) - 1;
  const int r_max = (m0 / rows != v_last / rows) ? rows - 1 : v_last % rows;
  const int kv_end = causal ? min(kv_len, ctx + r_max + 1) : kv_len;
  const int n_tiles = (kv_end + AN - 1) / AN;
  // global row of virtual row v in q [B, Hq, rows, hd]
  auto q_row = [&](int v) {
    return (static_cast<size_t>(b) * n_heads + hk * group + v / rows) * rows + v % rows;
  };

  constexpr int CPR = HD / 8;  // 16-byte chunks per Q / K row
  for (int i = tid; i < AM * CPR; i += 128) {
    const int r = i / CPR, c = i % CPR;
    const bool ok = m0 + r < n_virt;
    cp_async16(sQ + r * LD + c * 8, q + (ok ? q_row(m0 + r) : 0) * HD + c * 8, ok);
  }
  auto load_kv = [&](int t, int buf) {
    const int n0 = t * AN;
    for (int i = tid; i < AN * CPR; i += 128) {
      const int r = i / CPR, c = i % CPR;
      const bool ok = n0 + r < kv_end;
      cp_async16(sK + (buf * AN + r) * LD + c * 8, kb + static_cast<size_t>(ok ? n0 + r : 0) * HD + c * 8, ok);
    }
    if ((kv_stride & 7) == 0) {
      for (int i = tid; i < HD * (AN / 8); i += 128) {
        const int dd = i / (AN / 8), c = i % (AN / 8);
        const bool ok = n0 + c * 8 < kv_end;   // keys past kv_end inside a chunk get P = 0
        cp_async16(sV + (buf * HD + dd) * LDV + c * 8,
                   vb + static_cast<size_t>(dd) * kv_stride + (ok ? n0 + c * 8 : 0), ok);
      }
    } else {
      // rows of V^T are not 16-byte aligned: element loads, zeros past kv_end
      for (int i = tid; i < HD * AN; i += 128) {
        const int dd = i / AN, c = i % AN;
        sV[(buf * HD + dd) * LDV + c] =
            n0 + c < kv_end ? vb[static_cast<size_t>(dd) * kv_stride + n0 + c] : __float2bfloat16_rn(0.0f);
      }
    }
  };
  if (n_tiles > 0) load_kv(0, 0);
  cp_async_commit();

  float acc[HD / 8][4];
#pragma unroll
  for (int j = 0; j < HD / 8; ++j) acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.0f;
  float mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.0f, 0.0f};
  const int g = lane >> 2, t4 = lane & 3;
  // query positions of this lane's two fragment rows (virtual rows v and v + 8)
  const int v0 = m0 + warp * 16 + g;
  const int qpos_r[2] = {ctx + v0 % rows, ctx + (v0 + 8) % rows};
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
    const bf16* Vt = sV + buf * HD * LDV;
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
    const int n0 = t * AN;
    float tmax[2] = {-INFINITY, -INFINITY};
#pragma unroll
    for (int j = 0; j < AN / 8; ++j) {
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int key = n0 + j * 8 + 2 * t4 + (e & 1);
        const int qp = qpos_r[e >> 1];
        const bool ok = key < kv_end && (!causal || key < ctx || key <= qp) && (window <= 0 || qp - key < window);
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
    // O += P V, V^T tile [dim][key] is the col-major B operand
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
        const int dim = jj * 16 + (lane & 7) + (lane >> 4) * 8;
        const int key = kk * 16 + ((lane >> 3) & 1) * 8;
        ldsm_x4(vfr, Vt + dim * LDV + key);
        mma_bf16_16816(acc[2 * jj], pa, vfr[0], vfr[1]);
        mma_bf16_16816(acc[2 * jj + 1], pa, vfr[2], vfr[3]);
      }
    }
    __syncthreads();
  }
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 1);
    lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 2);
  }
  const size_t ldo = static_cast<size_t>(n_heads) * HD;
#pragma unroll
  for (int r = 0; r < 2; ++r) {
    const int v = v0 + r * 8;
    if (v >= n_virt) continue;
    const int row = v % rows, h = hk * group + v / rows;
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
                                                       const float* __restrict__ vt, float* __restrict__ o,
                                                       int n_heads, int n_kv_heads, int rows, int ctx,
                                                       int kv_stride, int causal, int window, float scale) {
  pdl_enter();
  constexpr int PL = HD / 32;
  const int lane = threadIdx.x & 31;
  const int row = blockIdx.x * 4 + (threadIdx.x >> 5);
  const int h = blockIdx.y, b = blockIdx.z;
  if (row >= rows) return;
  const int hk = h / (n_heads / n_kv_heads);
  const float* qr = q + ((static_cast<size_t>(b) * n_heads + h) * rows + row) * HD;
  const float* kb = k + (static_cast<size_t>(b) * n_kv_heads + hk) * kv_stride * HD;
  const float* vb = vt + (static_cast<size_t>(b) * n_kv_heads + hk) * HD * kv_stride;
  float qv[PL], acc[PL];
#pragma unroll
  for (int i = 0; i < PL; ++i) { qv[i] = qr[lane + 32 * i]; acc[i] = 0.0f; }
  const int qpos = ctx + row;
  const int kv_end = causal ? qpos + 1 : ctx + rows;
  const int kv_lo = window > 0 ? max(0, qpos - window + 1) : 0;   // sliding window start
  float m = -INFINITY, l = 0.0f;
  for (int j = kv_lo; j < kv_end; ++j) {
    float d = 0.0f;
#pragma unroll
    for (int i = 0; i < PL; ++i) d += qv[i] * kb[static_cast<size_t>(j) * HD + lane + 32 * i];
    d = warp_sum(d) * scale;
    const float mn = fmaxf(m, d);
    const float c = expf(m - mn), p = expf(d - mn);
    l = l * c + p;
#pragma unroll
    for (int i = 0; i < PL; ++i) acc[i] = acc[i] * c + p * vb[static_cast<size_t>(lane + 32 * i) * kv_stride + j];
    m = mn;
  }
  float* orow = o + (static_cast<size_t>(b) * rows + row) * n_heads * HD + static_cast<size_t>(h) * HD;
#pragma unroll
  for (int i = 0; i < PL; ++i) orow[lane + 32 * i] = acc[i] / l;
}

template <int HD>
cudaError_t launch_bf16(const AttnCall& a, cudaStream_t s) {
  const size_t smem = static_cast<size_t>(AM + 2 * AN) * (HD + 8) * sizeof(bf16) +
                      static_cast<size_t>(2 * HD) * (AN + 8) * sizeof(bf16);
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(attn_bf16_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    attr = true;
  }
  const int n_virt = (a.n_heads / a.n_kv_heads) * a.rows;
  dim3 grid((n_virt + AM - 1) / AM, a.n_kv_heads, a.batch);
  const float scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(HD));
  launch_pdl(attn_bf16_kernel<HD>, grid, 128, smem, s, static_cast<const bf16*>(a.q), static_cast<const bf16*>(a.k),
                                               static_cast<const bf16*>(a.v), static_cast<bf16*>(a.o), a.n_heads,
                                               a.n_kv_heads, a.rows, a.ctx, a.kv_stride, a.causal, a.window,
                                               scale_log2);
  return cudaGetLastError();
}

template <int HD>
cudaError_t launch_f32(const AttnCall& a, cudaStream_t s) {
  dim3 grid((a.rows + 3) / 4, a.n_heads, a.batch);
  launch_pdl(attn_f32_kernel<HD>, grid, 128, 0, s, static_cast<const float*>(a.q), static_cast<const float*>(a.k),
                                           static_cast<const float*>(a.v), static_cast<float*>(a.o), a.n_heads,
                                           a.n_kv_heads, a.rows, a.ctx, a.kv_stride, a.causal, a.window,
                                           1.0f / sqrtf(static_cast<float>(HD)));
  return cudaGetLastError();
}
}  // namespace

const char* attention(const AttnCall& a, cudaStream_t s) {
  if (a.rows <= 0 || a.batch <= 0) return nullptr;
  if (a.n_kv_heads <= 0 || a.n_heads % a.n_kv_heads) return "n_heads must be a multiple of n_kv_heads";
  if (a.kv_stride < a.ctx + a.rows) return "kv_stride smaller than ctx + rows";
  if (a.bf16) {
    // tcgen05 whenever the V^T rows are 16-byte aligned for TMA (the library's
    // KV buffers always are); 64-key tiles for hd 128 with few query rows
    const bool tc = a.kv_stride % 8 == 0 && (reinterpret_cast<uintptr_t>(a.q) & 15) == 0;
    if (a.head_dim == 64) {
      if (!tc) return launch_bf16<64>(a, s) == cudaSuccess ? nullptr : "attention launch failed";
      int dev = 0, n_sms = 0;
      cudaGetDevice(&dev);
      cudaDeviceGetAttribute(&n_sms, cudaDevAttrMultiProcessorCount, dev);
      const int ctas = ((a.n_heads / a.n_kv_heads) * a.rows + TQ - 1) / TQ * a.n_kv_heads * a.batch;
      const bool window_cuts = a.window > 0 && a.window < a.ctx + a.rows;
      if (attn_db_enabled() && !window_cuts && ctas > n_sms) return launch_db<64>(a, s);
      return launch_tc<64, 128>(a, s);
    }
    if (a.head_dim == 128) {
      if (!tc) return launch_bf16<128>(a, s) == cudaSuccess ? nullptr : "attention launch failed";
      // one CTA per SM: the pipelined kernel when the launch fills 80-100 % of the SMs in one wave (larger
      // launches run attn_tc_kernel two CTAs per SM, smaller ones split the keys)
      int dev = 0, n_sms = 0;
      cudaGetDevice(&dev);
      cudaDeviceGetAttribute(&n_sms, cudaDevAttrMultiProcessorCount, dev);
      const int ctas = ((a.n_heads / a.n_kv_heads) * a.rows + TQ - 1) / TQ * a.n_kv_heads * a.batch;
      const bool window_cuts = a.window > 0 && a.window < a.ctx + a.rows;
      if (attn_db_enabled() && !window_cuts && 5 * ctas >= 4 * n_sms && ctas <= n_sms) return launch_db<128>(a, s);
      return (a.n_heads / a.n_kv_heads) * a.rows < 2 * TQ ? launch_tc<128, 64>(a, s) : launch_tc<128, 128>(a, s);
    }
    return "bf16 attention supports head_dim 64 and 128";
  }
  cudaError_t e;
  if (a.head_dim == 32) e = launch_f32<32>(a, s);
  else if (a.head_dim == 64) e = launch_f32<64>(a, s);
  else if (a.head_dim == 128) e = launch_f32<128>(a, s);
  else return "fp32 attention supports head_dim 32, 64 and 128";
  return e == cudaSuccess ? nullptr : cudaGetErrorString(e);
}

}  // namespace tadm
