// bf16 GEMM on the 5th-generation tensor cores (tcgen05) for sm_103a.
//
//   acc[M, N] = A[M, K] * B[N, K]^T     (A, B bf16, K-major; fp32 accumulate)
//
// Persistent kernel, one CTA per SM, warp-specialised:
//   warp 0      one thread issues TMA loads of A / B tiles into a 4-stage
//               shared-memory ring (128-byte swizzle);
//   warp 1      allocates 512 TMEM columns (two 128 x 256 fp32 accumulators)
//               and one thread issues tcgen05.mma (M=128, N=256, K=16);
//   warps 2..9  epilogue: tcgen05.ld the accumulator rows (one TMEM lane per
//               thread; two warps per lane quadrant, each taking half of the
//               256 columns) and run the fused epilogue of epilogue.cuh, while
//               the MMA warp fills the other accumulator.
// GEMMs of more than 128 rows run the CTA-pair variant (gemm_tc2_kernel:
// 256 x 256 tiles, tcgen05.mma.cta_group::2, six stages), with split-K for
// the weight-streaming residual / fp32-store GEMMs whose tiles cannot fill
// the SMs; other GEMMs that need split-K run this kernel.
// Every mbarrier wait is bounded (mbar_wait_bounded): a role that gives up
// raises a shared abort flag and the device status word, and the CTA drains
// its in-flight copies and MMAs, frees TMEM and exits.
#include <cudaTypedefs.h>
#include <algorithm>
#include <cstdlib>
#include <mutex>

#include "epilogue.cuh"
#include "kernels.h"

namespace tadm {

namespace {
constexpr int BM = 128, BN = 256, BK = 64, STAGES = 4;
constexpr int A_BYTES = BM * BK * 2;   // 16 KB
constexpr int B_BYTES = BN * BK * 2;   // 32 KB
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int TMEM_COLS = 512;
constexpr int EPI_WARPS = 8;
constexpr int NUM_THREADS = 64 + 32 * EPI_WARPS;
constexpr int STAGE_OUT_BYTES = 32 * 128;   // per epilogue warp: 32 rows x 64 bf16
constexpr size_t SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + EPI_WARPS * STAGE_OUT_BYTES + 256;

// Accumulator rows of one warp (32 TMEM lanes) plus, when bf16 outputs are
// staged, the warp's 4 KB shared-memory box and the output tensor maps.
struct TmemSrc {
  static constexpr bool kStaged = true;
  uint32_t taddr;
  uint8_t* stage;                      // 32 rows x 128 B, 128-byte swizzle; null: direct stores
  const CUtensorMap* tm_out[2];
  int row0;                            // first of the warp's 32 output rows
  __device__ __forceinline__ bool staged() const { return stage != nullptr; }
  __device__ __forceinline__ bool has_box() const { return stage != nullptr; }
  // row `lane` of a 32 x 32 fp32 box (128-byte rows, 16-byte chunks XOR-swizzled by row)
  __device__ __forceinline__ void put_row(const float (&v)[32]) {
    const int lane = threadIdx.x & 31;
    __syncwarp();
    float4* row = reinterpret_cast<float4*>(stage + lane * 128);
#pragma unroll
    for (int q = 0; q < 8; ++q) row[q ^ (lane & 7)] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
    __syncwarp();
  }
  // element (row i, column lane) of that box
  __device__ __forceinline__ float get(int i) const {
    const int lane = threadIdx.x & 31;
    return reinterpret_cast<const float*>(stage + i * 128)[(((lane >> 2) ^ (i & 7)) << 2) | (lane & 3)];
  }
  __device__ __forceinline__ void load(int chunk, float (&v)[32]) {
    __syncwarp();  // tcgen05.ld is warp-collective: reconverge after divergent stores
    tmem_ld32(taddr + 32 * chunk, v);
  }
  // the same load without waiting: r is usable after wait_ld(r)
  __device__ __forceinline__ void load_async(int chunk, uint32_t (&r)[32]) {
    __syncwarp();
    tmem_ld32_nowait(taddr + 32 * chunk, r);
  }
  __device__ __forceinline__ void wait_ld(uint32_t (&r)[32]) { tmem_wait_ld(r); }
  // this lane's row of a 32 x 32 fp32 chunk into the box, then one TMA
  // reduce-add of the box into the fp32 output map at column x (resid += box)
  __device__ __forceinline__ void reduce32(int x, const float (&v)[32]) {
    const int lane = threadIdx.x & 31;
    if (lane == 0) bulk_wait_read0();   // the previous reduce has read the box
    put_row(v);
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
      tma_reduce_add_2d(tm_out[0], stage, x, row0);
      bulk_commit();
    }
  }
  // bf16 of a[0..31] and b[0..31] (output columns x .. x+63 of this lane's row)
  // into the box, then one TMA store of the warp's 32 x 64 block; rows and
  // columns outside the output are clipped by the tensor map.
  __device__ __forceinline__ void store64(int which, int x, const float (&a)[32], const float (&b)[32]) {
    const int lane = threadIdx.x & 31;
    if (lane == 0) bulk_wait_read0();   // the previous store has read the box
    __syncwarp();
    uint8_t* row = stage + lane * 128;
#pragma unroll
    for (int q = 0; q < 8; ++q) {
      const float* src = q < 4 ? &a[8 * q] : &b[8 * (q - 4)];
      __nv_bfloat162 t0 = __floats2bfloat162_rn(src[0], src[1]);
      __nv_bfloat162 t1 = __floats2bfloat162_rn(src[2], src[3]);
      __nv_bfloat162 t2 = __floats2bfloat162_rn(src[4], src[5]);
      __nv_bfloat162 t3 = __floats2bfloat162_rn(src[6], src[7]);
      *reinterpret_cast<uint4*>(row + ((q ^ (lane & 7)) << 4)) =
          make_uint4(*reinterpret_cast<uint32_t*>(&t0), *reinterpret_cast<uint32_t*>(&t1),
                     *reinterpret_cast<uint32_t*>(&t2), *reinterpret_cast<uint32_t*>(&t3));
    }
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
      tma_store_2d(tm_out[which], stage, x, row0);
      bulk_commit();
    }
  }
};

struct TcArgs {
  int M, N_acc, K;         // N_acc: accumulator columns in total (2F for GLU)
  int splits, kb_per_split;  // split-K: unit = (tile, K slice); partials [split][M][ldp] fp32
  float* part;
  size_t part_stride;
  int ldp;
  int staged;              // bf16 outputs go through the per-warp boxes and TMA stores
  int b_split;             // >0: B tile = 128 rows at n*128 and 128 rows at b_split + n*128
  int n_tiles_n;
  int kb_wrap;             // > 0: split hi + lo operand of kb_wrap k-blocks per half: k-block kb reads A's
                           // k-block (kb odd ? kb_wrap : 0) + kb / 2 and B's k-block kb / 2, so that the two
                           // reads of a B tile follow each other (the second one hits L2)
  int* status;
  const int* m_dev;        // optional device row count (<= M): tiles past it are skipped
  EpiParams ep;
};

// Tiles run N-fastest: the CTAs in flight share A tiles (activations, the
// large operand) through L2, and every weight matrix of the model fits in L2.
// At the start of a tile the producer asks L2 for the global rows its
// epilogue will read (residual stream, h, gate), so the epilogue does not wait
// on DRAM latency.
template <int EPI>
__device__ __forceinline__ void prefetch_epilogue_inputs(const TcArgs& a, int mb, int nb, int ncols = BN) {
  const EpiParams& p = a.ep;
  const float* src = nullptr;
  int ld = 0;
  if constexpr (EPI == EPI_RESID) { src = p.resid; ld = p.ldr; }
  else if constexpr (EPI == EPI_FUSION2 || EPI == EPI_ADD || EPI == EPI_PA_UP) { src = p.base; ld = p.ldb; }
  if (!src) return;
  const int n0 = nb * ncols, ncol = min(ncols, p.N - n0);
  if (ncol <= 0 || (ld & 3) || (n0 & 3)) return;
  const uint32_t bytes = static_cast<uint32_t>(ncol) * 4u & ~15u;
  for (int r = mb * BM; r < min(mb * BM + BM, p.M); ++r) prefetch_l2(src + static_cast<size_t>(r) * ld + n0, bytes);
}

template <int EPI>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmC, const __grid_constant__ CUtensorMap tmC2,
                   const TcArgs args) {
  pdl_enter();
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + STAGES * A_BYTES;
  uint8_t* sOut = smem + STAGES * STAGE_BYTES;          // EPI_WARPS boxes of 4 KB
  uint64_t* full = reinterpret_cast<uint64_t*>(sOut + EPI_WARPS * STAGE_OUT_BYTES);
  uint64_t* empty = full + STAGES;
  uint64_t* tfull = empty + STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], 32 * EPI_WARPS);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  const int m_run = args.m_dev ? min(args.M, *args.m_dev) : args.M;   // read after pdl_enter
  const int num_m = (m_run + BM - 1) / BM;
  const int tiles = num_m * args.n_tiles_n;
  const int units = tiles * args.splits;
  const int kblocks = (args.K + BK - 1) / BK;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------------------------------------------------------- producer
      int stage = 0;
      uint32_t phase = 0;
      int issued[STAGES];
      for (int s = 0; s < STAGES; ++s) issued[s] = 0;
      for (int unit = blockIdx.x; unit < units && !*abort_flag; unit += gridDim.x) {
        const int tile = unit / args.splits, ks = unit % args.splits;
        const int nb = tile % args.n_tiles_n, mb = tile / args.n_tiles_n;
        const int kb0 = ks * args.kb_per_split, kb1 = min(kblocks, kb0 + args.kb_per_split);
        if (args.splits == 1) prefetch_epilogue_inputs<EPI>(args, mb, nb);
        bool ok = true;
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait_bounded(&empty[stage], phase ^ 1, abort_flag, args.status)) { ok = false; break; }
          mbar_arrive_expect_tx(&full[stage], STAGE_BYTES);
          const int kba = args.kb_wrap > 0 ? (kb & 1) * args.kb_wrap + (kb >> 1) : kb;
          const int kbb = args.kb_wrap > 0 ? kb >> 1 : kb;
          tma_load_2d(sA + stage * A_BYTES, &tmA, &full[stage], kba * BK, mb * BM);
          if (args.b_split > 0) {
            tma_load_2d(sB + stage * B_BYTES, &tmB, &full[stage], kbb * BK, nb * (BN / 2));
            tma_load_2d(sB + stage * B_BYTES + B_BYTES / 2, &tmB, &full[stage], kbb * BK,
                        args.b_split + nb * (BN / 2));
          } else {
            tma_load_2d(sB + stage * B_BYTES, &tmB, &full[stage], kbb * BK, nb * BN);
          }
          ++issued[stage];
          if (++stage == STAGES) { stage = 0; phase ^= 1; }
        }
        if (!ok) break;
      }
      // every copy this thread started has landed before the CTA may exit
      for (int s = 0; s < STAGES; ++s)
        if (issued[s] > 0) {
          volatile int never = 0;
          mbar_wait_bounded(&full[s], (issued[s] - 1) & 1, &never, args.status);
        }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------------------------------------------------------- MMA issuer
      constexpr uint32_t idesc = idesc_bf16_f32(BM, BN);
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      for (int unit = blockIdx.x; unit < units && !*abort_flag; unit += gridDim.x) {
        const int ks = unit % args.splits;
        const int kb0 = ks * args.kb_per_split, kb1 = min(kblocks, kb0 + args.kb_per_split);
        if (!mbar_wait_bounded(&tempty[acc], acc_phase ^ 1, abort_flag, args.status)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * BN;
        bool ok = true;
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait_bounded(&full[stage], phase, abort_flag, args.status)) { ok = false; break; }
          tc_fence_after();
          const uint32_t a0 = smem_u32(sA + stage * A_BYTES);
          const uint32_t b0 = smem_u32(sB + stage * B_BYTES);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            umma_bf16(d_tmem, sdesc_kmajor_sw128(a0 + 32 * k), sdesc_kmajor_sw128(b0 + 32 * k), idesc,
                      (kb != kb0) || (k != 0));
          }
          umma_commit(&empty[stage]);
          if (++stage == STAGES) { stage = 0; phase ^= 1; }
        }
        if (!ok) break;
        umma_commit(&tfull[acc]);
        if (++acc == 2) { acc = 0; acc_phase ^= 1; }
      }
      // all MMAs issued by this thread are complete before TMEM is freed
      umma_commit(drain);
      volatile int never = 0;
      mbar_wait_bounded(drain, 0, &never, args.status);
    }
  } else {
    // ------------------------------------------------------------------ epilogue
    const int quad = warp & 3;               // TMEM lanes 32*quad .. 32*quad+31 (hardware rule)
    const int part = (warp - 2) / 4;         // which half of the columns
    constexpr int nsplit = EPI == EPI_PA_GATE ? 1 : 2;
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int unit = blockIdx.x; unit < units; unit += gridDim.x) {
      if (!warp_wait_bounded(&tfull[acc], acc_phase, abort_flag, args.status)) break;
      tc_fence_after();
      const int tile = unit / args.splits, ks = unit % args.splits;
      const int nb = tile % args.n_tiles_n, mb = tile / args.n_tiles_n;
      TmemSrc src{tmem_base + static_cast<uint32_t>(acc * BN) + (static_cast<uint32_t>(quad * 32) << 16),
                  args.staged ? sOut + (warp - 2) * STAGE_OUT_BYTES : nullptr, {&tmC, &tmC2}, mb * BM + quad * 32};
      const int m = mb * BM + quad * 32 + lane;
      if (args.splits > 1) {
        // raw fp32 partial of this K slice, tile-local column order
        float v[32];
        float* dst = args.part + ks * args.part_stride + static_cast<size_t>(m) * args.ldp + nb * BN;
        for (int c = part * (BN / 64); c < (part + 1) * (BN / 64); ++c) {
          src.load(c, v);
          if (m < args.M) store32(dst, 0, 32 * c, v, 32);
        }
      } else if (part < nsplit) {
        epilogue_row<EPI>(args.ep, m, nb, BN, src, part, nsplit);
      }
      tc_fence_before();
      mbar_arrive(&tempty[acc]);
      if (++acc == 2) { acc = 0; acc_phase ^= 1; }
    }
    if (args.staged && lane == 0) bulk_wait0();   // every TMA store of this warp (if any) is complete
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

// ------------------------------------------------------- CTA-pair variant
// One 256 x 256 tile per 2-CTA cluster with tcgen05.mma.cta_group::2 (M=256,
// N=256, K=16): CTA r holds A rows 128r..128r+127 of the tile and B rows
// 128r..128r+127 (its half of the N columns) in its own shared memory, and
// its 128 rows of the accumulator in its own TMEM.  Each SM thus receives
// 32 KB of operands per 64-deep k-block instead of 48 KB for the same MMA
// work, and six stages fit in shared memory.  Roles per CTA as above; only
// the even CTA's MMA thread issues.  Barriers: both producers count their
// bytes on the even CTA's full[s] (the even producer expects both CTAs'
// bytes); the MMA thread's commits release empty[s] and signal tfull[a] in
// both CTAs; every epilogue warp of both CTAs releases an accumulator on the
// even CTA's tempty[a].
// PBN: columns of the pair tile (256, or 128 for GEMMs whose 256-wide pair
// tiles would leave most SMs idle).
template <int PBN>
struct PairCfg {
  static constexpr int STAGES = PBN == 256 ? 6 : 8;
  static constexpr int A_BYTES = BM * BK * 2;            // 16 KB
  static constexpr int B_BYTES = (PBN / 2) * BK * 2;     // this CTA's half of B: 16 KB / 8 KB
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr size_t SMEM = 1024 + STAGES * STAGE_BYTES + EPI_WARPS * STAGE_OUT_BYTES + 256;
  static_assert(SMEM <= 232448, "pair GEMM shared memory");
};

template <int EPI, int PBN>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(NUM_THREADS, 1)
    gemm_tc2_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                    const __grid_constant__ CUtensorMap tmC, const __grid_constant__ CUtensorMap tmC2,
                    const TcArgs args) {
  pdl_enter();
  using PC = PairCfg<PBN>;
  constexpr int P_STAGES = PC::STAGES, P_A_BYTES = PC::A_BYTES, P_B_BYTES = PC::B_BYTES;
  constexpr int P_STAGE_BYTES = PC::STAGE_BYTES;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + P_STAGES * P_A_BYTES;
  uint8_t* sOut = smem + P_STAGES * P_STAGE_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(sOut + EPI_WARPS * STAGE_OUT_BYTES);
  uint64_t* empty = full + P_STAGES;
  uint64_t* tfull = empty + P_STAGES;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  if (threadIdx.x == 0) {
    for (int s = 0; s < P_STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], 2 * EPI_WARPS);   // one arrival per epilogue warp of either CTA
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmB);
  }
  if (warp == 1) {
    tmem_alloc_pair(tmem_slot, TMEM_COLS);   // one warp of each CTA, collectively
    tmem_relinquish_pair();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();   // the peer's barriers are initialised (and its TMEM allocated) before any signal
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  const int m_run = args.m_dev ? min(args.M, *args.m_dev) : args.M;   // read after pdl_enter
  const int num_m2 = (m_run + 2 * BM - 1) / (2 * BM);
  const int units = num_m2 * args.n_tiles_n * args.splits;   // unit = (pair tile, K slice)
  const int u0 = static_cast<int>(blockIdx.x >> 1), ustep = static_cast<int>(gridDim.x >> 1);
  const int kblocks = (args.K + BK - 1) / BK;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------------------------------------------------------- producer (both CTAs)
      const uint32_t full_l0 = cluster_addr(full, 0);   // the even CTA's full[0]
      int stage = 0;
      uint32_t phase = 0;
      for (int unit = u0; unit < units && !*abort_flag; unit += ustep) {
        const int tile = unit / args.splits, ks = unit % args.splits;
        const int nb = tile % args.n_tiles_n;
        const int mb = 2 * (tile / args.n_tiles_n) + static_cast<int>(rank);   // this CTA's 128-row block
        const int kb0 = ks * args.kb_per_split, kb1 = min(kblocks, kb0 + args.kb_per_split);
        if (args.splits == 1) prefetch_epilogue_inputs<EPI>(args, mb, nb, PBN);
        const int brow = args.b_split > 0 ? (rank ? args.b_split : 0) + nb * (PBN / 2) : nb * PBN + rank * (PBN / 2);
        bool ok = true;
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait_bounded(&empty[stage], phase ^ 1, abort_flag, args.status)) { ok = false; break; }
          if (leader) mbar_arrive_expect_tx(&full[stage], 2 * P_STAGE_BYTES);
          const uint32_t fb = full_l0 + 8u * stage;
          const int kba = args.kb_wrap > 0 ? (kb & 1) * args.kb_wrap + (kb >> 1) : kb;
          const int kbb = args.kb_wrap > 0 ? kb >> 1 : kb;
          tma_load_2d_pair(sA + stage * P_A_BYTES, &tmA, fb, kba * BK, mb * BM);
          tma_load_2d_pair(sB + stage * P_B_BYTES, &tmB, fb, kbb * BK, brow);
          if (++stage == P_STAGES) { stage = 0; phase ^= 1; }
        }
        if (!ok) break;
      }
      // the MMA thread's last commits arrive on these barriers (from the even
      // CTA): wait until every stage is released, which also means every copy
      // into this CTA's shared memory has landed and been consumed
      for (int i = 0; i < P_STAGES; ++i) {
        mbar_wait_bounded(&empty[stage], phase ^ 1, abort_flag, args.status);
        if (++stage == P_STAGES) { stage = 0; phase ^= 1; }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && leader) {
      // ---------------------------------------------------------------- MMA issuer (even CTA)
      constexpr uint32_t idesc = idesc_bf16_f32(2 * BM, PBN);
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      for (int unit = u0; unit < units && !*abort_flag; unit += ustep) {
        const int ks = unit % args.splits;
        const int kb0 = ks * args.kb_per_split, kb1 = min(kblocks, kb0 + args.kb_per_split);
        if (!mbar_wait_bounded(&tempty[acc], acc_phase ^ 1, abort_flag, args.status)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * PBN;
        bool ok = true;
        for (int kb = kb0; kb < kb1; ++kb) {
          if (!mbar_wait_bounded(&full[stage], phase, abort_flag, args.status)) { ok = false; break; }
          tc_fence_after();
          const uint32_t a0 = smem_u32(sA + stage * P_A_BYTES);
          const uint32_t b0 = smem_u32(sB + stage * P_B_BYTES);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            umma_bf16_pair(d_tmem, sdesc_kmajor_sw128(a0 + 32 * k), sdesc_kmajor_sw128(b0 + 32 * k), idesc,
                           (kb != kb0) || (k != 0));
          }
          umma_commit_pair_mc(&empty[stage], 0x3);
          if (++stage == P_STAGES) { stage = 0; phase ^= 1; }
        }
        if (!ok) break;
        umma_commit_pair_mc(&tfull[acc], 0x3);
        if (++acc == 2) { acc = 0; acc_phase ^= 1; }
      }
      // every pair MMA is complete (both CTAs' TMEM written) before TMEM is freed
      umma_commit_pair_mc(drain, 0x1);
      volatile int never = 0;
      mbar_wait_bounded(drain, 0, &never, args.status);
    }
  } else {
    // ------------------------------------------------------------------ epilogue (both CTAs)
    const int quad = warp & 3;
    const int part = (warp - 2) / 4;
    constexpr int nsplit = EPI == EPI_PA_GATE ? 1 : 2;
    const uint32_t tempty_l0 = cluster_addr(tempty, 0);
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int unit = u0; unit < units; unit += ustep) {
      if (!warp_wait_bounded(&tfull[acc], acc_phase, abort_flag, args.status)) break;
      tc_fence_after();
      const int tile = unit / args.splits, ks = unit % args.splits;
      const int nb = tile % args.n_tiles_n;
      const int mb = 2 * (tile / args.n_tiles_n) + static_cast<int>(rank);
      TmemSrc src{tmem_base + static_cast<uint32_t>(acc * PBN) + (static_cast<uint32_t>(quad * 32) << 16),
                  args.staged ? sOut + (warp - 2) * STAGE_OUT_BYTES : nullptr, {&tmC, &tmC2}, mb * BM + quad * 32};
      const int m = mb * BM + quad * 32 + lane;
      if (args.splits > 1) {
        // raw fp32 partial of this K slice: this CTA's 128 rows of the pair tile, columns in natural order
        if (mb * BM < args.M) {
          float v[32];
          float* dst = args.part + ks * args.part_stride + static_cast<size_t>(m) * args.ldp + nb * PBN;
          for (int c = part * (PBN / 64); c < (part + 1) * (PBN / 64); ++c) {
            src.load(c, v);
            if (m < args.M) store32(dst, 0, 32 * c, v, 32);
          }
        }
      } else if (part < nsplit && mb * BM < args.M) {   // the odd CTA's rows may lie past M
        epilogue_row<EPI>(args.ep, m, nb, PBN, src, part, nsplit);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_remote(tempty_l0 + 8u * acc);
      if (++acc == 2) { acc = 0; acc_phase ^= 1; }
    }
    if (args.staged && lane == 0) bulk_wait0();
  }

  tc_fence_before();
  __syncthreads();
  // neither CTA frees TMEM or exits while the pair's MMAs, copies or
  // barrier signals may still reach it
  cluster_sync();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, TMEM_COLS);
  }
}

// --------------------------------------------------------------------- host
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;
int g_num_sms = 0;
bool g_pair_mma = true;   // CTA-pair kernel for large GEMMs; TADM_GEMM_PAIRS=0 keeps every GEMM on one CTA per tile

bool get_encoder() {
  std::call_once(g_encode_once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&g_num_sms, cudaDevAttrMultiProcessorCount, dev);
    const char* env = getenv("TADM_GEMM_PAIRS");
    if (env && env[0] == '0') g_pair_mma = false;
  });
  return g_encode != nullptr;
}

// 2-D bf16 tensor map over rows x cols (row stride ld elements), box of
// box_rows x 64 elements, 128-byte swizzle, zero fill out of bounds.
bool make_map(CUtensorMap* m, const void* ptr, int64_t rows, int64_t cols, int64_t ld, int box_rows) {
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld * 2)};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(BK), static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// 2-D fp32 map over rows x cols (row stride ld elements), box 32 rows x 32, 128-byte swizzle.
bool make_f32_map(CUtensorMap* m, const void* ptr, int64_t rows, int64_t cols, int64_t ld) {
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld * 4)};
  cuuint32_t box[2] = {32, 32};
  cuuint32_t estr[2] = {1, 1};
  return g_encode(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<void*>(ptr), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 2-D bf16 output map over rows x cols (row stride ld), box 32 rows x 64, 128-byte swizzle.
bool make_out_map(CUtensorMap* m, const void* ptr, int64_t rows, int64_t cols, int64_t ld) {
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld * 2)};
  cuuint32_t box[2] = {64, 32};
  cuuint32_t estr[2] = {1, 1};
  return g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int EPI>
cudaError_t launch_epi(const CUtensorMap& ta, const CUtensorMap& tb, const CUtensorMap& tc, const CUtensorMap& tc2,
                       const TcArgs& a, int grid, cudaStream_t s) {
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(gemm_tc_kernel<EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(SMEM_BYTES));
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  launch_pdl(gemm_tc_kernel<EPI>, grid, NUM_THREADS, SMEM_BYTES, s, ta, tb, tc, tc2, a);
  return cudaGetLastError();
}

// CTA-pair kernel: `pairs` = 256-row x 256-column tiles; the grid is capped at
// the number of 2-CTA clusters that fit on the GPU at once (a persistent grid
// larger than that would run its last clusters after the others).
template <int EPI, int PBN = 256>
cudaError_t launch_epi_pair(const CUtensorMap& ta, const CUtensorMap& tb, const CUtensorMap& tc,
                            const CUtensorMap& tc2, const TcArgs& a, int pairs, cudaStream_t s) {
  constexpr size_t smem = PairCfg<PBN>::SMEM;
  static int max_clusters = 0;
  if (max_clusters == 0) {
    cudaError_t e = cudaFuncSetAttribute(gemm_tc2_kernel<EPI, PBN>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(g_num_sms & ~1);
    cfg.blockDim = dim3(NUM_THREADS);
    cfg.dynamicSmemBytes = smem;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, gemm_tc2_kernel<EPI, PBN>, &cfg) != cudaSuccess || n <= 0) {
      cudaGetLastError();
      n = g_num_sms / 2;
    }
    max_clusters = n;
  }
  const int clusters = std::min(pairs, max_clusters);
  launch_pdl(gemm_tc2_kernel<EPI, PBN>, 2 * clusters, NUM_THREADS, smem, s, ta, tb, tc, tc2, a);
  return cudaGetLastError();
}

}  // namespace

const char* gemm_tc(const GemmCall& g, cudaStream_t s) {
  if (!get_encoder()) return "cuTensorMapEncodeTiled is unavailable";
  if (g.M <= 0 || g.N <= 0 || g.K <= 0) return nullptr;
  if (g.K % 8 || g.lda % 8 || g.ldb % 8) return "bf16 GEMM needs K, lda, ldb multiples of 8";
  if (g.k_b > 0 && (g.K != 2 * g.k_b || g.k_b % BK)) return "split operand GEMM needs K = 2 k_b, k_b % 64 == 0";
  const int k_b = g.k_b > 0 ? g.k_b : g.K;   // columns of B
  if ((reinterpret_cast<uintptr_t>(g.A) | reinterpret_cast<uintptr_t>(g.B)) & 15)
    return "bf16 GEMM operands must be 16-byte aligned";
  const bool glu = g.epi == EPI_GLU;
  CUtensorMap ta, tb;
  if (!make_map(&ta, g.A, g.A_rows > 0 ? g.A_rows : g.M, g.K, g.lda, BM)) return "tensor map (A) encode failed";
  const int64_t b_rows = glu ? 2LL * g.N : g.N;
  if (!make_map(&tb, g.B, b_rows, k_b, g.ldb, glu ? BN / 2 : BN)) return "tensor map (B) encode failed";
  TcArgs a;
  a.M = g.M;
  a.K = g.K;
  a.N_acc = glu ? 2 * g.N : g.N;
  a.b_split = glu ? g.N : 0;
  a.n_tiles_n = glu ? (g.N + BN / 2 - 1) / (BN / 2) : (g.N + BN - 1) / BN;
  a.kb_wrap = g.k_b > 0 ? g.k_b / BK : 0;
  if (glu && g.N % (BN / 2)) return "GLU GEMM needs the FFN width to be a multiple of 128";
  if (g.epi == EPI_QKV && BN % g.ep.head_dim) return "head_dim must divide 256";
  if (g.epi == EPI_PA_GATE && g.N > BN) return "gate GEMM needs N <= 256";
  a.status = g.status;
  a.m_dev = g.m_dev;
  a.ep = g.ep;
  a.ep.M = g.M;
  a.ep.N = g.N;
  a.ep.n_tiles = a.n_tiles_n * (g.epi == EPI_LMHEAD ? 2 : 1);   // one partial per column half
  // bf16 outputs of the plain, GLU and fusion-gate epilogues go out through TMA stores
  CUtensorMap tc{}, tc2{};
  a.staged = 0;
  auto aligned = [](const void* p, int ld) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0 && ld % 8 == 0; };
  a.ep.resid_tma = 0;
  if (g.epi == EPI_RESID || g.epi == EPI_FUSION2) {
    a.staged = 1;   // the boxes serve as transpose scratch, or as the source of TMA reduce-adds
    if (g.epi == EPI_RESID && (reinterpret_cast<uintptr_t>(g.ep.resid) & 15) == 0 && g.ep.ldr % 4 == 0 &&
        make_f32_map(&tc, g.ep.resid, g.M, g.N, g.ep.ldr))
      a.ep.resid_tma = 1;
  } else if (g.ep.out_bf16 && (g.epi == EPI_STORE || g.epi == EPI_GLU)) {
    if (aligned(g.ep.out, g.ep.ldo) && make_out_map(&tc, g.ep.out, g.M, g.N, g.ep.ldo)) a.staged = 1;
  } else if (g.ep.out_bf16 && g.epi == EPI_FUSION1 && g.ep.d_split % 64 == 0) {
    if (aligned(g.ep.out, g.ep.ldo) && aligned(g.ep.out2, g.ep.ldo2) &&
        make_out_map(&tc, g.ep.out, g.M, g.ep.d_split, g.ep.ldo) &&
        make_out_map(&tc2, g.ep.out2, g.M, g.N - g.ep.d_split, g.ep.ldo2))
      a.staged = 1;
  }
  const int tiles = ((g.M + BM - 1) / BM) * a.n_tiles_n;
  // split-K when the tiles cannot fill the SMs and K is long: fixed-order
  // reduction afterwards, so results do not depend on the split
  const int kblocks = (g.K + BK - 1) / BK;
  a.splits = 1;
  a.kb_per_split = kblocks;
  a.ldp = a.n_tiles_n * BN;
  // CTA-pair tiles that keep >= 40% of the SMs busy beat split-K: no fp32
  // partials, no reduction launches.  Residual, fusion-output and QKV GEMMs
  // whose 256-wide pair tiles would occupy at most half the SMs (the
  // weight-streaming block steps) use 256 x 128 pair tiles instead.
  const int m_pairs = (g.M + 2 * BM - 1) / (2 * BM);
  const bool pair_ok = g_pair_mma && g.M > BM;
  const bool narrow_kind = g.epi == EPI_RESID || g.epi == EPI_FUSION2 || (g.epi == EPI_QKV && 128 % g.ep.head_dim == 0);
  const bool narrow = pair_ok && narrow_kind && m_pairs * a.n_tiles_n * 4 <= g_num_sms;
  const int pair_units = narrow ? m_pairs * ((g.N + 127) / 128) : m_pairs * a.n_tiles_n;
  // pairs must keep >= 40% of the SMs busy to beat split-K; for the residual-add and fp32-store epilogues,
  // whose split-K reduction is one element-wise launch, >= 60% (the weight-streaming block steps)
  const bool elem_reduce = g.epi == EPI_RESID || (g.epi == EPI_STORE && !g.ep.out_bf16);
  const bool pairs_fill = pair_ok && 2 * pair_units * (elem_reduce ? 10 : 5) >= g_num_sms * (elem_reduce ? 6 : 2);
  // The residual-add / fp32-store GEMMs whose 256 x 256 pair tiles fill under
  // 60 % of the SMs take those tiles with split-K: each weight tile crosses
  // L2 once (128 x 256 tiles fetch it once per 128-row block) and an SM
  // receives 32 KB per k-block (256 x 128 pair tiles: 24 KB for half the MMA
  // work; 128 x 256 tiles: 48 KB for the same work).
  const bool wide_fill = 2 * m_pairs * a.n_tiles_n * 10 >= g_num_sms * 6;
  if (pair_ok && elem_reduce && !wide_fill && g.split_buf && !g.m_dev && kblocks >= 8) {
    const int pu = m_pairs * a.n_tiles_n;
    int sp = std::min(std::min((g_num_sms / 2) / pu, kblocks / 4), 16);
    const size_t per = static_cast<size_t>(g.M) * a.ldp * sizeof(float);
    while (sp > 1 && sp * per > g.split_bytes) --sp;
    if (sp > 1) {
      CUtensorMap tbh;
      if (!make_map(&tbh, g.B, b_rows, k_b, g.ldb, BN / 2)) return "tensor map (B, half tiles) encode failed";
      TcArgs a2 = a;
      a2.kb_per_split = (kblocks + sp - 1) / sp;
      a2.splits = (kblocks + a2.kb_per_split - 1) / a2.kb_per_split;
      a2.part = g.split_buf;
      a2.part_stride = static_cast<size_t>(g.M) * a2.ldp;
      a2.staged = 0;
      const cudaError_t e = g.epi == EPI_RESID ? launch_epi_pair<EPI_RESID>(ta, tbh, tc, tc2, a2, pu * a2.splits, s)
                                               : launch_epi_pair<EPI_STORE>(ta, tbh, tc, tc2, a2, pu * a2.splits, s);
      if (e != cudaSuccess) return cudaGetErrorString(e);
      const_cast<GemmCall&>(g).launched = 1;
      int nr = 0;
      const char* r = splitk_reduce(g.epi, a2.ep, a2.part, a2.part_stride, a2.ldp, a2.splits, a2.n_tiles_n, s, &nr);
      if (r) return r;
      const_cast<GemmCall&>(g).launched = 1 + nr;
      return nullptr;
    }
  }
  // QKV GEMMs of the same regime (whose 256 x 128 pair tiles re-read the
  // activation operand once per cluster) likewise: 256-wide pair tiles with
  // split-K; the QKV epilogue (QK-norm, RoPE, Q / K / V writes) runs in the
  // split-K reduction on the slice-ordered sum.
  if (narrow && g.epi == EPI_QKV && g.split_buf && !g.m_dev && kblocks >= 16) {
    const int pu = m_pairs * a.n_tiles_n;
    int sp = std::min(std::min((g_num_sms / 2) / pu, kblocks / 8), 16);
    const size_t per = static_cast<size_t>(g.M) * a.ldp * sizeof(float);
    while (sp > 1 && sp * per > g.split_bytes) --sp;
    if (sp > 1) {
      CUtensorMap tbh;
      if (!make_map(&tbh, g.B, b_rows, k_b, g.ldb, BN / 2)) return "tensor map (B, half tiles) encode failed";
      TcArgs a2 = a;
      a2.kb_per_split = (kblocks + sp - 1) / sp;
      a2.splits = (kblocks + a2.kb_per_split - 1) / a2.kb_per_split;
      a2.part = g.split_buf;
      a2.part_stride = static_cast<size_t>(g.M) * a2.ldp;
      a2.staged = 0;
      const cudaError_t e = launch_epi_pair<EPI_QKV>(ta, tbh, tc, tc2, a2, pu * a2.splits, s);
      if (e != cudaSuccess) return cudaGetErrorString(e);
      const_cast<GemmCall&>(g).launched = 1;
      int nr = 0;
      const char* r = splitk_reduce(g.epi, a2.ep, a2.part, a2.part_stride, a2.ldp, a2.splits, a2.n_tiles_n, s, &nr);
      if (r) return r;
      const_cast<GemmCall&>(g).launched = 1 + nr;
      return nullptr;
    }
  }
  if (g.split_buf && !g.m_dev && !pairs_fill && tiles * 3 < g_num_sms * 2 && kblocks >= 8) {
    int sp = std::min(std::min(g_num_sms / tiles, kblocks / 4), 16);
    const size_t per = static_cast<size_t>(g.M) * a.ldp * sizeof(float);
    while (sp > 1 && sp * per > g.split_bytes) --sp;
    if (sp > 1) {
      a.kb_per_split = (kblocks + sp - 1) / sp;
      a.splits = (kblocks + a.kb_per_split - 1) / a.kb_per_split;
      a.part = g.split_buf;
      a.part_stride = static_cast<size_t>(g.M) * a.ldp;
      a.staged = 0;
    }
  }
  // CTA pairs (256 x 256 tiles, cta_group::2) for every unsplit GEMM of more
  // than 128 rows: the same SMs as 128 x 256 tiles, less operand traffic each
  if (pair_ok && a.splits == 1 && narrow) {
    CUtensorMap tbh;
    if (!make_map(&tbh, g.B, b_rows, k_b, g.ldb, 64)) return "tensor map (B, quarter tiles) encode failed";
    TcArgs a2 = a;
    a2.n_tiles_n = (g.N + 127) / 128;
    cudaError_t e = g.epi == EPI_RESID  ? launch_epi_pair<EPI_RESID, 128>(ta, tbh, tc, tc2, a2, pair_units, s)
                    : g.epi == EPI_QKV  ? launch_epi_pair<EPI_QKV, 128>(ta, tbh, tc, tc2, a2, pair_units, s)
                                        : launch_epi_pair<EPI_FUSION2, 128>(ta, tbh, tc, tc2, a2, pair_units, s);
    if (e != cudaSuccess) return cudaGetErrorString(e);
    const_cast<GemmCall&>(g).launched = 1;
    return nullptr;
  }
  if (pair_ok && a.splits == 1) {
    CUtensorMap tbh;
    if (!make_map(&tbh, g.B, b_rows, k_b, g.ldb, BN / 2)) return "tensor map (B, half tiles) encode failed";
    cudaError_t e;
    switch (g.epi) {
      case EPI_STORE: e = launch_epi_pair<EPI_STORE>(ta, tbh, tc, tc2, a, pair_units, s); break;
      case EPI_RESID: e = launch_epi_pair<EPI_RESID>(ta, tbh, tc, tc2, a, pair_units, s); break;
      case EPI_QKV: e = launch_epi_pair<EPI_QKV>(ta, tbh, tc, tc2, a, pair_units, s); break;
      case EPI_GLU: e = launch_epi_pair<EPI_GLU>(ta, tbh, tc, tc2, a, pair_units, s); break;
      case EPI_FUSION1: e = launch_epi_pair<EPI_FUSION1>(ta, tbh, tc, tc2, a, pair_units, s); break;
      case EPI_FUSION2: e = launch_epi_pair<EPI_FUSION2>(ta, tbh, tc, tc2, a, pair_units, s); break;
      case EPI_LMHEAD: e = launch_epi_pair<EPI_LMHEAD>(ta, tbh, tc, tc2, a, pair_units, s); break;
      case EPI_PA_UP: e = launch_epi_pair<EPI_PA_UP>(ta, tbh, tc, tc2, a, pair_units, s); break;
      case EPI_SILU: e = launch_epi_pair<EPI_SILU>(ta, tbh, tc, tc2, a, pair_units, s); break;
      case EPI_ADD: e = launch_epi_pair<EPI_ADD>(ta, tbh, tc, tc2, a, pair_units, s); break;
      case EPI_PA_GATE: e = launch_epi_pair<EPI_PA_GATE>(ta, tbh, tc, tc2, a, pair_units, s); break;
      default: return "unknown epilogue";
    }
    if (e != cudaSuccess) return cudaGetErrorString(e);
    const_cast<GemmCall&>(g).launched = 1;
    return nullptr;
  }
  const int units = tiles * a.splits;
  const int grid = units < g_num_sms ? units : g_num_sms;
  cudaError_t e;
  switch (g.epi) {
    case EPI_STORE: e = launch_epi<EPI_STORE>(ta, tb, tc, tc2, a, grid, s); break;
    case EPI_RESID: e = launch_epi<EPI_RESID>(ta, tb, tc, tc2, a, grid, s); break;
    case EPI_QKV: e = launch_epi<EPI_QKV>(ta, tb, tc, tc2, a, grid, s); break;
    case EPI_GLU: e = launch_epi<EPI_GLU>(ta, tb, tc, tc2, a, grid, s); break;
    case EPI_FUSION1: e = launch_epi<EPI_FUSION1>(ta, tb, tc, tc2, a, grid, s); break;
    case EPI_FUSION2: e = launch_epi<EPI_FUSION2>(ta, tb, tc, tc2, a, grid, s); break;
    case EPI_LMHEAD: e = launch_epi<EPI_LMHEAD>(ta, tb, tc, tc2, a, grid, s); break;
    case EPI_PA_UP: e = launch_epi<EPI_PA_UP>(ta, tb, tc, tc2, a, grid, s); break;
    case EPI_SILU: e = launch_epi<EPI_SILU>(ta, tb, tc, tc2, a, grid, s); break;
    case EPI_ADD: e = launch_epi<EPI_ADD>(ta, tb, tc, tc2, a, grid, s); break;
    case EPI_PA_GATE: e = launch_epi<EPI_PA_GATE>(ta, tb, tc, tc2, a, grid, s); break;
    default: return "unknown epilogue";
  }
  if (e != cudaSuccess) return cudaGetErrorString(e);
  const_cast<GemmCall&>(g).launched = 1;
  if (a.splits > 1) {
    int nr = 0;
    const char* r = splitk_reduce(g.epi, a.ep, a.part, a.part_stride, a.ldp, a.splits, a.n_tiles_n, s, &nr);
    if (r) return r;
    const_cast<GemmCall&>(g).launched = 1 + nr;
  }
  return nullptr;
}

size_t gemm_tc_split_bytes() {
  get_encoder();
  return static_cast<size_t>(g_num_sms > 0 ? g_num_sms : 160) * BM * BN * sizeof(float);
}

int gemm_tc_tiles_n(int N, int epi) {
  if (epi == EPI_LMHEAD) return 2 * ((N + 255) / 256);   // partials: one per half tile
  return epi == EPI_GLU ? (N + 127) / 128 : (N + 255) / 256;
}

}  // namespace tadm
