// Loss contraction on the 5th-generation tensor cores (sm_103a):
//   G[e] = alpha * D[e] H[e]^T   (bf16 operands, fp32 accumulation in TMEM)
// D[e] is R x C row-major, H[e] is C x C row-major and symmetric, so both are
// "K-major" operands (the contraction index is contiguous) and H^T = H gives
// G = 2 D H_sym = dL/dW^ of L = tr(D H D^T) (Eq. 1 with a linear layer).
//
// Two persistent, warp-specialised kernels: k_tc_gemm (one CTA per SM, below)
// and k_tc_gemm_pair (CTA pairs sharing one cta_group::2 MMA, the default; see
// its own comment).  k_tc_gemm:
//   warp 0     TMA producer: 128x64 tile of D and BNx64 tile of H per stage
//              (BN = 128, 224 or 256), 128-byte swizzle, into a ring of as many
//              stages as shared memory holds;
//   warp 1     TMEM allocator and MMA issuer: tcgen05.mma.cta_group::1.kind::f16
//              M=128 N=BN K=16, four per 64-wide k-block, accumulating in TMEM;
//              tcgen05.commit frees a stage / publishes a finished accumulator;
//   warps 2-5  epilogue: tcgen05.ld 32x32b of the accumulator (each warp owns
//              the 32 TMEM lanes of its quarter), scale by alpha, store fp32.
// The accumulator is double-buffered in TMEM (2 x BN columns) so the epilogue
// of tile i overlaps the MMAs of tile i+1.  Every mbarrier wait is bounded
// (2 s of %globaltimer); on expiry the CTA records an error code in the
// workspace flags, waits (bounded) for its own in-flight copies, frees its TMEM
// and returns.
#include <cuda.h>
#include <cuda_bf16.h>

#include "gsq_internal.h"
#include "gsq_tc.cuh"

namespace gsq {

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn get_encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

bool encode_kmajor_bf16(CUtensorMap* map, const void* base, uint64_t inner, uint64_t rows,
                        uint32_t box_rows) {
  EncodeTiledFn fn = get_encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[2] = {inner, rows};
  const cuuint64_t strides[1] = {inner * 2};
  const cuuint32_t box[2] = {64u, box_rows};  // 64 bf16 = one 128-byte swizzle row
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Output of the CTA-pair GEMM as a 3D map [E][M][N] (fp32 or bf16) for TMA
// stores of 32 x 32 boxes, swizzled 128 B (fp32 rows) or 64 B (bf16 rows).
static bool encode_out_map(CUtensorMap* map, void* base, int E, int M, int N, int bf16) {
  EncodeTiledFn fn = get_encode_fn();
  if (!fn) return false;
  const uint64_t es = bf16 ? 2 : 4;
  const cuuint64_t dims[3] = {static_cast<cuuint64_t>(N), static_cast<cuuint64_t>(M),
                              static_cast<cuuint64_t>(E)};
  const cuuint64_t strides[2] = {static_cast<cuuint64_t>(N) * es,
                                 static_cast<cuuint64_t>(M) * N * es};
  const cuuint32_t box[3] = {32u, 32u, 1u};
  const cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, bf16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, base,
            dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
            bf16 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

namespace {

constexpr int TC_BM = 128, TC_BK = 64;
constexpr int TC_A_BYTES = TC_BM * TC_BK * 2;
constexpr int TC_THREADS = 192;

// Tile shape M = 128 x N = BN (256, 224 or 128) x 64; the pipeline fills the shared memory.
template <int BN>
struct TcCfg {
  static constexpr int kBBytes = BN * TC_BK * 2;
  static constexpr int kStageBytes = TC_A_BYTES + kBBytes;
  // as many stages as the 227 KiB of shared memory per CTA hold (barriers + 1 KiB
  // alignment slack beside them), at most 8
  static constexpr int kStages =
      ((232448 - 2048) / kStageBytes) < 8 ? ((232448 - 2048) / kStageBytes) : 8;
  // double-buffered fp32 accumulator (2 BN columns), allocated as a power of two
  static constexpr int kTmemCols = 2 * BN <= 256 ? 256 : 512;
  static constexpr int kAccStride = kTmemCols / 2;  // column offset of the second buffer
  static constexpr int kSmemBytes = kStages * kStageBytes + 256 + 1024;
  // kind::f16 instruction descriptor: D fp32 (bits 4-5 = 1), A bf16 (7-9 = 1),
  // B bf16 (10-12 = 1), both K-major (bits 15, 16 = 0), N>>3 at 17-22, M>>4 at 24-28.
  static constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) |
                                     (static_cast<uint32_t>(BN >> 3) << 17) |
                                     (static_cast<uint32_t>(TC_BM >> 4) << 24);
};

struct TcArgs {
  int stall;      // test hook: skip the first k-block's copies, so the waits on it run out
  int E, M, N, K;
  int group_n;    // tile-order column group (tile_coords)
  void* out;      // [E][M][N], fp32 or bf16
  int out_bf16;
  float alpha;
  DevFlags* flags;
  int sym_per_e;  // > 0: symmetric output, only the upper-triangle tiles (tile_coords_upper)
};

// Output tile `tile` of the launch: the full order of tile_coords, or the upper
// triangle of a symmetric output.
__device__ __forceinline__ void tile_at(const TcArgs& a, int tile, int Mt, int Nt, int BM, int BN,
                                        int& e, int& m, int& n) {
  if (a.sym_per_e > 0)
    tile_coords_upper(tile, Mt, Nt, BM, BN, a.sym_per_e, e, m, n);
  else
    tile_coords(tile, Mt, Nt, a.group_n, e, m, n);
}

template <int BN>
__global__ void __launch_bounds__(TC_THREADS, 1)
    k_tc_gemm(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
              const TcArgs args) {
  constexpr int TC_BN = BN;
  constexpr int TC_STAGES = TcCfg<BN>::kStages;
  constexpr int TC_STAGE_BYTES = TcCfg<BN>::kStageBytes;
  constexpr int TC_TMEM_COLS = TcCfg<BN>::kTmemCols;
  constexpr uint32_t TC_IDESC = TcCfg<BN>::kIdesc;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint64_t* full_bar = reinterpret_cast<uint64_t*>(smem + TC_STAGES * TC_STAGE_BYTES);
  uint64_t* empty_bar = full_bar + TC_STAGES;
  uint64_t* tfull_bar = empty_bar + TC_STAGES;
  uint64_t* tempty_bar = tfull_bar + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty_bar + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < TC_STAGES; ++s) {
      mbar_init(full_bar + s, 1);
      mbar_init(empty_bar + s, 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(tfull_bar + a, 1);
      mbar_init(tempty_bar + a, 128);
    }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmA)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmB)) : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_slot)),
                 "r"(TC_TMEM_COLS));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  grid_dep_wait();  // A, B and the output may belong to the stream's previous kernel until here
  grid_dep_launch();

  const int Mt = (args.M + TC_BM - 1) / TC_BM;
  const int Nt = (args.N + TC_BN - 1) / TC_BN;
  const int KB = (args.K + TC_BK - 1) / TC_BK;
  static_assert(TC_STAGES >= 2, "pipeline depth");
  const int tiles = args.E * (args.sym_per_e > 0 ? args.sym_per_e : Mt * Nt);

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      int stage = 0;
      uint32_t phase = 0;
      uint32_t issued_phase[TC_STAGES];
      bool issued[TC_STAGES];
      for (int s = 0; s < TC_STAGES; ++s) issued[s] = false;
      bool ok = true;
      for (int tile = blockIdx.x; ok && tile < tiles; tile += gridDim.x) {
        int e, m, n;
        tile_at(args, tile, Mt, Nt, TC_BM, TC_BN, e, m, n);
        const int arow = e * args.M + m * TC_BM;
        const int brow = e * args.N + n * TC_BN;
        for (int kb = 0; kb < KB; ++kb) {
          if (!mbar_wait(empty_bar + stage, phase ^ 1u, abort_flag)) {
            ok = false;
            break;
          }
          uint8_t* sa = smem + stage * TC_STAGE_BYTES;
          uint8_t* sb = sa + TC_A_BYTES;
          if (!(args.stall && tile == static_cast<int>(blockIdx.x) && kb == 0)) {
            mbar_expect_tx(full_bar + stage, TC_STAGE_BYTES);
            tma_load_2d(sa, &tmA, full_bar + stage, kb * TC_BK, arow);
            tma_load_2d(sb, &tmB, full_bar + stage, kb * TC_BK, brow);
            issued[stage] = true;
            issued_phase[stage] = phase;
          }
          if (++stage == TC_STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok) {
        // abort: wait (bounded, ignoring the abort flag) for our own copies in flight
        for (int s = 0; s < TC_STAGES; ++s)
          if (issued[s]) mbar_wait(full_bar + s, issued_phase[s], abort_flag, false);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true;
      for (int tile = blockIdx.x; ok && tile < tiles; tile += gridDim.x) {
        if (!mbar_wait(tempty_bar + acc, acc_phase ^ 1u, abort_flag)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * TcCfg<BN>::kAccStride);
        for (int kb = 0; kb < KB; ++kb) {
          if (!mbar_wait(full_bar + stage, phase, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + stage * TC_STAGE_BYTES);
          const uint64_t da = sw128_desc(sa);
          const uint64_t db = sw128_desc(sa + TC_A_BYTES);
#pragma unroll
          for (int k = 0; k < TC_BK / 16; ++k)  // advance 16 bf16 = 32 B = 2 units of 16 B
            umma_bf16(d_tmem, da + 2 * k, db + 2 * k, TC_IDESC, (kb | k) != 0 ? 1u : 0u);
          umma_commit(empty_bar + stage);
          if (++stage == TC_STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        umma_commit(tfull_bar + acc);
        if (++acc == 2) {
          acc = 0;
          acc_phase ^= 1u;
        }
      }
    }
  } else {
    // ---------------- epilogue (warps 2..5) ----------------
    const int quarter = warp & 3;  // TMEM lanes 32*quarter .. +31 are this warp's
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int tile = blockIdx.x; tile < tiles; tile += gridDim.x) {
      if (!mbar_wait(tfull_bar + acc, acc_phase, abort_flag)) break;
      tc_fence_after();
      int e, m, n;
      tile_at(args, tile, Mt, Nt, TC_BM, TC_BN, e, m, n);
      const int row = m * TC_BM + quarter * 32 + lane;
      const int col0 = n * TC_BN;
      const int64_t obase = (static_cast<int64_t>(e) * args.M + row) * args.N;
      const uint32_t taddr = tmem_base + static_cast<uint32_t>(acc * TcCfg<BN>::kAccStride) +
                             (static_cast<uint32_t>(quarter * 32) << 16);
#pragma unroll 1
      for (int c = 0; c < TC_BN; c += 16) {
        float v[16];
        tmem_ld16(taddr + c, v);
        if (row < args.M) {
#pragma unroll
          for (int j = 0; j < 16; j += 4) {
            const int col = col0 + c + j;
            if (col < args.N) {
              const float4 o = make_float4(args.alpha * v[j], args.alpha * v[j + 1],
                                           args.alpha * v[j + 2], args.alpha * v[j + 3]);
              if (args.out_bf16) {
                const __nv_bfloat162 lo = __floats2bfloat162_rn(o.x, o.y);
                const __nv_bfloat162 hi = __floats2bfloat162_rn(o.z, o.w);
                uint2 raw;
                raw.x = *reinterpret_cast<const uint32_t*>(&lo);
                raw.y = *reinterpret_cast<const uint32_t*>(&hi);
                *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(args.out) + obase + col) = raw;
              } else {
                *reinterpret_cast<float4*>(static_cast<float*>(args.out) + obase + col) = o;
              }
            }
          }
        }
      }
      tc_fence_before();
      mbar_arrive(tempty_bar + acc);
      if (++acc == 2) {
        acc = 0;
        acc_phase ^= 1u;
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base),
                 "r"(TC_TMEM_COLS));
  }
  if (threadIdx.x == 0 && *abort_flag) atomicExch(&args.flags->error, 0x7C01u);
}

// ---------------------------------------------------------------------------
// CTA-pair variant: a cluster of two CTAs on neighbouring SMs computes a
// 256 x BN output tile with tcgen05.mma.cta_group::2.  Each CTA stages its own
// 128 rows of A and its half (BN/2 rows) of B, so a stage is 16 KiB + BN KiB/8
// (30 KiB at BN = 224, 6 stages beside 32 KiB of epilogue staging) and every
// SM streams a third less operand data than a single CTA with the same tile
// width.  Both CTAs' copies complete on the leader's (rank 0) full barrier; the
// leader's single MMA thread issues for the pair and its commits arrive on the
// empty / accumulator barriers of both CTAs.  Each CTA's epilogue drains its
// own TMEM (its 128 rows) through shared memory into TMA tensor stores and
// arrives on the leader's accumulator-empty barrier.  Waits are bounded as in
// k_tc_gemm; a CTA that gives up records the error, lets its copies in flight
// land (a bounded pause) and meets its peer at the final cluster barrier.
// ---------------------------------------------------------------------------
constexpr int TC2_BM = 256;  // rows per pair tile (128 per CTA)

template <int BN>
struct Tc2Cfg {
  static constexpr int kBHalf = BN / 2;
  static constexpr int kBBytes = kBHalf * TC_BK * 2;
  static constexpr int kStageBytes = TC_A_BYTES + kBBytes;
  // epilogue staging: two 32 x 32 fp32 chunks per epilogue warp (4 warps)
  static constexpr int kEpiChunk = 32 * 32 * 4;
  static constexpr int kEpiBytes = 4 * 2 * kEpiChunk;
  static constexpr int kStages =
      ((232448 - 2048 - kEpiBytes) / kStageBytes) < 8 ? ((232448 - 2048 - kEpiBytes) / kStageBytes)
                                                       : 8;
  static constexpr int kTmemCols = 2 * BN <= 256 ? 256 : 512;
  static constexpr int kAccStride = kTmemCols / 2;
  static constexpr int kSmemBytes = kStages * kStageBytes + kEpiBytes + 256 + 1024;
  static constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) |
                                     (static_cast<uint32_t>(BN >> 3) << 17) |
                                     (static_cast<uint32_t>(TC2_BM >> 4) << 24);
  static_assert(BN % 32 == 0, "the epilogue stores 32-column chunks");
  static_assert(kBHalf % 8 == 0, "B half must be whole 8-row swizzle atoms");
  static_assert(kStageBytes % 1024 == 0, "stages must keep 1 KiB alignment");
};

template <int BN>
__global__ void __launch_bounds__(TC_THREADS, 1)
    k_tc_gemm_pair(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmO, const TcArgs args) {
  using Cfg = Tc2Cfg<BN>;
  constexpr int STAGES = Cfg::kStages;
  constexpr int STAGE_BYTES = Cfg::kStageBytes;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* epi = smem + STAGES * STAGE_BYTES;  // epilogue staging (1 KiB aligned)
  uint64_t* full_bar = reinterpret_cast<uint64_t*>(epi + Cfg::kEpiBytes);
  uint64_t* empty_bar = full_bar + STAGES;
  uint64_t* tfull_bar = empty_bar + STAGES;
  uint64_t* tempty_bar = tfull_bar + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty_bar + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();  // 0: leader, 1: peer
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full_bar + s, 1);
      mbar_init(empty_bar + s, 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(tfull_bar + a, 1);
      mbar_init(tempty_bar + a, 8);  // one arrival per epilogue warp of both CTAs
    }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmA)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmB)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmO)) : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_slot)),
                 "r"(Cfg::kTmemCols));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // both CTAs' barriers exist before any copy or arrival reaches them
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  grid_dep_wait();  // A, B and the output may belong to the stream's previous kernel until here
  grid_dep_launch();

  const int Mt = (args.M + TC2_BM - 1) / TC2_BM;
  const int Nt = (args.N + BN - 1) / BN;
  const int KB = (args.K + TC_BK - 1) / TC_BK;
  const int tiles = args.E * (args.sym_per_e > 0 ? args.sym_per_e : Mt * Nt);
  const int pair = blockIdx.x >> 1, npairs = gridDim.x >> 1;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer (both CTAs) ----------------
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int tile = pair; ok && tile < tiles; tile += npairs) {
        int e, m, n;
        tile_at(args, tile, Mt, Nt, TC2_BM, BN, e, m, n);
        const int arow = e * args.M + m * TC2_BM + static_cast<int>(rank) * TC_BM;
        const int brow = e * args.N + n * BN + static_cast<int>(rank) * Cfg::kBHalf;
        for (int kb = 0; kb < KB; ++kb) {
          if (!mbar_wait(empty_bar + stage, phase ^ 1u, abort_flag)) {
            ok = false;
            break;
          }
          uint8_t* sa = smem + stage * STAGE_BYTES;
          uint8_t* sb = sa + TC_A_BYTES;
          const uint32_t fb = mapa_shared(smem_u32(full_bar + stage), 0);
          if (!(args.stall && tile == pair && kb == 0)) {
            if (rank == 0) mbar_expect_tx(full_bar + stage, 2 * STAGE_BYTES);
            tma_load_2d_pair(sa, &tmA, fb, kb * TC_BK, arow);
            tma_load_2d_pair(sb, &tmB, fb, kb * TC_BK, brow);
          }
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok) {
        // copies in flight complete on the leader's barrier: give them time to land
        const unsigned long long t0 = global_ns();
        while (global_ns() - t0 < 200000ull) __nanosleep(1000);
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && rank == 0) {
      // ---------------- MMA issuer (leader only, for the pair) ----------------
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true;
      for (int tile = pair; ok && tile < tiles; tile += npairs) {
        if (!mbar_wait(tempty_bar + acc, acc_phase ^ 1u, abort_flag)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * Cfg::kAccStride);
        for (int kb = 0; kb < KB; ++kb) {
          if (!mbar_wait(full_bar + stage, phase, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + stage * STAGE_BYTES);
          const uint64_t da = sw128_desc(sa);
          const uint64_t db = sw128_desc(sa + TC_A_BYTES);
#pragma unroll
          for (int k = 0; k < TC_BK / 16; ++k)
            umma_bf16_pair(d_tmem, da + 2 * k, db + 2 * k, Cfg::kIdesc, (kb | k) != 0 ? 1u : 0u);
          umma_commit_pair(empty_bar + stage);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        umma_commit_pair(tfull_bar + acc);
        if (++acc == 2) {
          acc = 0;
          acc_phase ^= 1u;
        }
      }
    }
  } else {
    // ---------------- epilogue (warps 2..5 of both CTAs) ----------------
    // Each warp drains its 32 TMEM lanes (rows) 32 columns at a time into one of
    // two 32 x 32 staging chunks and writes the chunk with one TMA tensor store
    // (whole-line writes).  The store map is 3D [E][M][N], so rows past M of an
    // expert and columns past N are not written.  Staging layout = the map's
    // swizzle (128 B for fp32 rows, 64 B for bf16 rows): 16-byte piece p of row r
    // sits at piece p ^ (r % 8) (fp32) or p ^ ((r / 2) % 4) (bf16), so the 32
    // lanes' writes of one piece spread over all banks.
    const int quarter = warp & 3;
    uint8_t* wbuf = epi + quarter * 2 * Cfg::kEpiChunk;
    int acc = 0;
    uint32_t acc_phase = 0;
    int chunks = 0;  // chunks this warp has stored; buffer = chunks & 1
    for (int tile = pair; tile < tiles; tile += npairs) {
      if (!mbar_wait(tfull_bar + acc, acc_phase, abort_flag)) break;
      tc_fence_after();
      int e, m, n;
      tile_at(args, tile, Mt, Nt, TC2_BM, BN, e, m, n);
      const int row0 = m * TC2_BM + static_cast<int>(rank) * TC_BM + quarter * 32;
      const int col0 = n * BN;
      const uint32_t taddr = tmem_base + static_cast<uint32_t>(acc * Cfg::kAccStride) +
                             (static_cast<uint32_t>(quarter * 32) << 16);
#pragma unroll 1
      for (int c = 0; c < BN; c += 32) {
        float v[32];
        tmem_ld32(taddr + c, v);
        if (row0 >= args.M || col0 + c >= args.N) continue;  // nothing of this chunk is stored
        uint8_t* buf = wbuf + (chunks & 1) * Cfg::kEpiChunk;
        if (chunks >= 2) {  // the store that last read this buffer has finished reading it
          if (lane == 0) bulk_wait_read_1();
          __syncwarp();
        }
        if (args.out_bf16) {
          uint8_t* rowp = buf + lane * 64;
          const int sw = (lane >> 1) & 3;
#pragma unroll
          for (int p = 0; p < 4; ++p) {
            uint32_t w[4];
#pragma unroll
            for (int h = 0; h < 4; ++h) {
              const __nv_bfloat162 b2 = __floats2bfloat162_rn(args.alpha * v[8 * p + 2 * h],
                                                              args.alpha * v[8 * p + 2 * h + 1]);
              w[h] = *reinterpret_cast<const uint32_t*>(&b2);
            }
            *reinterpret_cast<uint4*>(rowp + 16 * (p ^ sw)) = make_uint4(w[0], w[1], w[2], w[3]);
          }
        } else {
          uint8_t* rowp = buf + lane * 128;
          const int sw = lane & 7;
#pragma unroll
          for (int p = 0; p < 8; ++p)
            *reinterpret_cast<float4*>(rowp + 16 * (p ^ sw)) =
                make_float4(args.alpha * v[4 * p], args.alpha * v[4 * p + 1],
                            args.alpha * v[4 * p + 2], args.alpha * v[4 * p + 3]);
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          tma_store_3d(&tmO, buf, col0 + c, row0, e);
          bulk_commit();
        }
        ++chunks;
        // Pace the drain over the next tile's MMAs: drained back to back, the staging
        // writes and store reads of a whole accumulator slowed the tensor pipe
        // (measured on GB300, 4096^3: 88.4 us back to back, 87.2 us with 600 ns
        // between chunks, 87.7 us with 1.5 us).  Not after this CTA's last tile.
        if (tile + npairs < tiles) __nanosleep(600);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(mapa_shared(smem_u32(tempty_bar + acc), 0));
      if (++acc == 2) {
        acc = 0;
        acc_phase ^= 1u;
      }
    }
    if (lane == 0) bulk_wait_all();  // every store complete before the CTA leaves
    __syncwarp();
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync();  // neither CTA leaves while the pair's MMAs or arrivals may touch it
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem_base),
                 "r"(Cfg::kTmemCols));
  }
  if (threadIdx.x == 0 && *abort_flag) atomicExch(&args.flags->error, 0x7C04u);
}

// ---------------------------------------------------------------------------
// Clusters of two CTA pairs (four CTAs) on the same column tile and adjacent
// 256-row tiles: pair p of the cluster (cluster ranks 2p, 2p + 1) computes row
// tile 2 mc + p, both pairs column tile n.  Both pairs need the same BN rows of
// B, so each CTA loads a quarter of them (BN/4 rows) and multicasts it to the
// CTA of the other pair that holds the same half: CTA (p, q) loads rows
// q BN/2 + p BN/4 .. + BN/4 into both CTAs (0, q) and (1, q) at the matching
// offset of their B half.  A (each pair's own rows) is loaded as in
// k_tc_gemm_pair.  An SM then requests 16 KiB + BN/4 x 128 B per k-block from
// L2 instead of 16 KiB + BN/2 x 128 B.  Barriers: each pair's full barrier (in
// its leader) counts the bytes landing in both its CTAs, whichever CTA issued
// them; a stage is free again only when both pairs' MMAs have read it (the
// empty barriers take one commit from each pair's leader, multicast to all
// four CTAs); accumulator barriers stay per pair.  Waits are bounded as in
// k_tc_gemm_pair; a CTA that gives up records 0x7C05.
// ---------------------------------------------------------------------------
template <int BN>
__global__ void __launch_bounds__(TC_THREADS, 1)
    k_tc_gemm_quad(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmBq,
                   const __grid_constant__ CUtensorMap tmO, const TcArgs args) {
  using Cfg = Tc2Cfg<BN>;
  constexpr int STAGES = Cfg::kStages;
  constexpr int STAGE_BYTES = Cfg::kStageBytes;
  constexpr int BQ = BN / 4;  // rows of B each CTA loads and multicasts
  static_assert(BQ % 8 == 0, "B quarters must be whole 8-row swizzle atoms");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* epi = smem + STAGES * STAGE_BYTES;
  uint64_t* full_bar = reinterpret_cast<uint64_t*>(epi + Cfg::kEpiBytes);
  uint64_t* empty_bar = full_bar + STAGES;
  uint64_t* tfull_bar = empty_bar + STAGES;
  uint64_t* tempty_bar = tfull_bar + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty_bar + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t crank = cluster_ctarank();   // 0..3
  const uint32_t pp = crank >> 1;             // pair within the cluster
  const uint32_t q = crank & 1u;              // CTA within the pair (0: leader)
  const uint32_t leader = crank & ~1u;
  const uint16_t pair_mask = static_cast<uint16_t>(3u << (2 * pp));
  const uint16_t half_mask = static_cast<uint16_t>((1u << q) | (1u << (q + 2)));
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full_bar + s, 1);
      mbar_init(empty_bar + s, 2);  // one commit from each pair's leader
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(tfull_bar + a, 1);
      mbar_init(tempty_bar + a, 8);  // one arrival per epilogue warp of the pair
    }
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmA)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmBq)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmO)) : "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_slot)),
                 "r"(Cfg::kTmemCols));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // every CTA's barriers exist before any copy or arrival reaches them
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  grid_dep_wait();  // A, B and the output may belong to the stream's previous kernel until here
  grid_dep_launch();

  const int Mt = (args.M + TC2_BM - 1) / TC2_BM;
  const int Mt2 = (Mt + 1) / 2;  // row-tile pairs per expert
  const int Nt = (args.N + BN - 1) / BN;
  const int KB = (args.K + TC_BK - 1) / TC_BK;
  const int tiles = args.E * Mt2 * Nt;  // cluster tiles
  const int cl = blockIdx.x >> 2, ncl = gridDim.x >> 2;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer (every CTA) ----------------
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      const uint32_t fb_base = mapa_shared(smem_u32(full_bar), leader);
      for (int tile = cl; ok && tile < tiles; tile += ncl) {
        int e, mc, n;
        tile_coords(tile, Mt2, Nt, args.group_n, e, mc, n);
        const int m = 2 * mc + static_cast<int>(pp);
        const int arow = e * args.M + m * TC2_BM + static_cast<int>(q) * TC_BM;
        const int brow = e * args.N + n * BN + static_cast<int>(q) * Cfg::kBHalf +
                         static_cast<int>(pp) * BQ;
        for (int kb = 0; kb < KB; ++kb) {
          if (!mbar_wait(empty_bar + stage, phase ^ 1u, abort_flag)) {
            ok = false;
            break;
          }
          uint8_t* sa = smem + stage * STAGE_BYTES;
          uint8_t* sbq = sa + TC_A_BYTES + pp * (BQ * TC_BK * 2);
          const uint32_t fb = fb_base + static_cast<uint32_t>(stage * sizeof(uint64_t));
          if (!(args.stall && tile == cl && kb == 0)) {
            if (q == 0) mbar_expect_tx(full_bar + stage, 2 * STAGE_BYTES);
            tma_load_2d_pair(sa, &tmA, fb, kb * TC_BK, arow);
            tma_load_2d_pair_mc(sbq, &tmBq, fb, kb * TC_BK, brow, half_mask);
          }
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok) {
        const unsigned long long t0 = global_ns();
        while (global_ns() - t0 < 200000ull) __nanosleep(1000);
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && q == 0) {
      // ---------------- MMA issuer (each pair's leader) ----------------
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      bool ok = true;
      for (int tile = cl; ok && tile < tiles; tile += ncl) {
        if (!mbar_wait(tempty_bar + acc, acc_phase ^ 1u, abort_flag)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * Cfg::kAccStride);
        for (int kb = 0; kb < KB; ++kb) {
          if (!mbar_wait(full_bar + stage, phase, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + stage * STAGE_BYTES);
          const uint64_t da = sw128_desc(sa);
          const uint64_t db = sw128_desc(sa + TC_A_BYTES);
#pragma unroll
          for (int k = 0; k < TC_BK / 16; ++k)
            umma_bf16_pair(d_tmem, da + 2 * k, db + 2 * k, Cfg::kIdesc, (kb | k) != 0 ? 1u : 0u);
          umma_commit_mask(empty_bar + stage, 0xF);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        umma_commit_mask(tfull_bar + acc, pair_mask);
        if (++acc == 2) {
          acc = 0;
          acc_phase ^= 1u;
        }
      }
    }
  } else {
    // ---------------- epilogue (warps 2..5 of every CTA), as in k_tc_gemm_pair ------------
    const int quarter = warp & 3;
    uint8_t* wbuf = epi + quarter * 2 * Cfg::kEpiChunk;
    int acc = 0;
    uint32_t acc_phase = 0;
    int chunks = 0;
    const uint32_t te_base = mapa_shared(smem_u32(tempty_bar), leader);
    for (int tile = cl; tile < tiles; tile += ncl) {
      if (!mbar_wait(tfull_bar + acc, acc_phase, abort_flag)) break;
      tc_fence_after();
      int e, mc, n;
      tile_coords(tile, Mt2, Nt, args.group_n, e, mc, n);
      const int m = 2 * mc + static_cast<int>(pp);
      const int row0 = m * TC2_BM + static_cast<int>(q) * TC_BM + quarter * 32;
      const int col0 = n * BN;
      const uint32_t taddr = tmem_base + static_cast<uint32_t>(acc * Cfg::kAccStride) +
                             (static_cast<uint32_t>(quarter * 32) << 16);
#pragma unroll 1
      for (int c = 0; c < BN; c += 32) {
        float v[32];
        tmem_ld32(taddr + c, v);
        if (m >= Mt || row0 >= args.M || col0 + c >= args.N) continue;  // nothing of it is stored
        uint8_t* buf = wbuf + (chunks & 1) * Cfg::kEpiChunk;
        if (chunks >= 2) {
          if (lane == 0) bulk_wait_read_1();
          __syncwarp();
        }
        if (args.out_bf16) {
          uint8_t* rowp = buf + lane * 64;
          const int sw = (lane >> 1) & 3;
#pragma unroll
          for (int p = 0; p < 4; ++p) {
            uint32_t w[4];
#pragma unroll
            for (int h = 0; h < 4; ++h) {
              const __nv_bfloat162 b2 = __floats2bfloat162_rn(args.alpha * v[8 * p + 2 * h],
                                                              args.alpha * v[8 * p + 2 * h + 1]);
              w[h] = *reinterpret_cast<const uint32_t*>(&b2);
            }
            *reinterpret_cast<uint4*>(rowp + 16 * (p ^ sw)) = make_uint4(w[0], w[1], w[2], w[3]);
          }
        } else {
          uint8_t* rowp = buf + lane * 128;
          const int sw = lane & 7;
#pragma unroll
          for (int p = 0; p < 8; ++p)
            *reinterpret_cast<float4*>(rowp + 16 * (p ^ sw)) =
                make_float4(args.alpha * v[4 * p], args.alpha * v[4 * p + 1],
                            args.alpha * v[4 * p + 2], args.alpha * v[4 * p + 3]);
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          tma_store_3d(&tmO, buf, col0 + c, row0, e);
          bulk_commit();
        }
        ++chunks;
        if (tile + ncl < tiles) __nanosleep(600);  // pace the drain (k_tc_gemm_pair)
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(te_base + static_cast<uint32_t>(acc * sizeof(uint64_t)));
      if (++acc == 2) {
        acc = 0;
        acc_phase ^= 1u;
      }
    }
    if (lane == 0) bulk_wait_all();
    __syncwarp();
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync();  // no CTA leaves while the cluster's MMAs, copies or arrivals may touch it
  if (warp == 1) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem_base),
                 "r"(Cfg::kTmemCols));
  }
  if (threadIdx.x == 0 && *abort_flag) atomicExch(&args.flags->error, 0x7C05u);
}

bool tc_supported_impl(int device) {
  cudaDeviceProp prop;
  if (cudaGetDeviceProperties(&prop, device) != cudaSuccess) return false;
  return prop.major == 10 && prop.minor == 3 && get_encode_fn() != nullptr;
}

// Fraction of the last wave's SMs that have a tile: tiles / (waves * SMs).
double wave_balance(int64_t tiles, int num_sms) {
  const int64_t waves = (tiles + num_sms - 1) / num_sms;
  return static_cast<double>(tiles) / static_cast<double>(waves * num_sms);
}

// Tiles of one expert's upper triangle (tile_coords_upper) for an M x M output in
// BM x BN tiles.
int upper_tiles(int M, int BM, int BN) {
  const int Mt = (M + BM - 1) / BM, Nt = (M + BN - 1) / BN;
  int count = 0;
  for (int m = 0; m < Mt; ++m) count += Nt - (m * BM) / BN;
  return count;
}

template <int BN>
cudaError_t launch_tc_gemm_bn(const TcGemm& g, int num_sms, cudaStream_t s) {
  // set on every launch: the attribute belongs to the current device
  cudaError_t ea = cudaFuncSetAttribute(k_tc_gemm<BN>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                        TcCfg<BN>::kSmemBytes);
  if (ea != cudaSuccess) return ea;
  CUtensorMap ta, tb;
  if (g.K % 8 != 0 || g.N % 4 != 0) return cudaErrorInvalidValue;  // 16-B rows; 8/16-B stores
  if (!encode_kmajor_bf16(&ta, g.A, static_cast<uint64_t>(g.K),
                          static_cast<uint64_t>(g.E) * g.M, TC_BM) ||
      !encode_kmajor_bf16(&tb, g.B, static_cast<uint64_t>(g.K),
                          static_cast<uint64_t>(g.E) * g.N, BN))
    return cudaErrorInvalidValue;
  TcArgs a;
  a.E = g.E;
  a.M = g.M;
  a.N = g.N;
  a.K = g.K;
  a.group_n = g.group_n > 0 ? g.group_n : (g.N + BN - 1) / BN;
  a.out = g.out;
  a.out_bf16 = g.out_bf16;
  a.alpha = g.alpha;
  a.flags = g.flags;
  a.stall = g.stall;
  a.sym_per_e = g.sym ? upper_tiles(g.M, TC_BM, BN) : 0;
  const int Mt = (g.M + TC_BM - 1) / TC_BM, Nt = (g.N + BN - 1) / BN;
  const int64_t tiles = static_cast<int64_t>(g.E) * (g.sym ? a.sym_per_e : Mt * Nt);
  const int grid = static_cast<int>(tiles < num_sms ? tiles : num_sms);
  cudaLaunchAttribute attr[1];
  pdl_attr(attr[0]);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid, 1, 1);
  cfg.blockDim = dim3(TC_THREADS, 1, 1);
  cfg.dynamicSmemBytes = TcCfg<BN>::kSmemBytes;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = g.pdl ? 1 : 0;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, k_tc_gemm<BN>, ta, tb, a);
  return e != cudaSuccess ? e : cudaGetLastError();
}

template <int BN>
cudaError_t launch_tc_gemm_pair_bn(const TcGemm& g, int num_sms, cudaStream_t s) {
  using Cfg = Tc2Cfg<BN>;
  // set on every launch: the attribute belongs to the current device
  cudaError_t ea = cudaFuncSetAttribute(k_tc_gemm_pair<BN>,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kSmemBytes);
  if (ea != cudaSuccess) return ea;
  CUtensorMap ta, tb, to;
  if (g.K % 8 != 0 || g.N % 4 != 0) return cudaErrorInvalidValue;
  if (g.out_bf16 && g.N % 8 != 0) return cudaErrorInvalidValue;  // 16-byte row pitch of the store map
  if ((reinterpret_cast<uintptr_t>(g.out) & 15) != 0) return cudaErrorInvalidValue;
  if (!encode_kmajor_bf16(&ta, g.A, static_cast<uint64_t>(g.K),
                          static_cast<uint64_t>(g.E) * g.M, TC_BM) ||
      !encode_kmajor_bf16(&tb, g.B, static_cast<uint64_t>(g.K),
                          static_cast<uint64_t>(g.E) * g.N, Cfg::kBHalf) ||
      !encode_out_map(&to, g.out, g.E, g.M, g.N, g.out_bf16))
    return cudaErrorInvalidValue;
  TcArgs a;
  a.E = g.E;
  a.M = g.M;
  a.N = g.N;
  a.K = g.K;
  a.group_n = g.group_n > 0 ? g.group_n : (g.N + BN - 1) / BN;
  a.out = g.out;
  a.out_bf16 = g.out_bf16;
  a.alpha = g.alpha;
  a.flags = g.flags;
  a.stall = g.stall;
  a.sym_per_e = g.sym ? upper_tiles(g.M, TC2_BM, BN) : 0;
  const int Mt = (g.M + TC2_BM - 1) / TC2_BM, Nt = (g.N + BN - 1) / BN;
  const int64_t tiles = static_cast<int64_t>(g.E) * (g.sym ? a.sym_per_e : Mt * Nt);
  int pairs = num_sms / 2;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  pdl_attr(attr[1]);
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.blockDim = dim3(TC_THREADS, 1, 1);
  cfg.dynamicSmemBytes = Cfg::kSmemBytes;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cfg.gridDim = dim3(2 * pairs, 1, 1);
  int max_clusters = 0;
  if (cudaOccupancyMaxActiveClusters(&max_clusters, k_tc_gemm_pair<BN>, &cfg) != cudaSuccess ||
      max_clusters < 1) {
    cudaGetLastError();
    return launch_tc_gemm_bn<BN>(g, num_sms, s);  // no CTA pair can be resident: single CTAs
  }
  if (max_clusters < pairs) pairs = max_clusters;
  if (tiles < pairs) pairs = static_cast<int>(tiles);
  cfg.gridDim = dim3(2 * pairs, 1, 1);
  cfg.numAttrs = g.pdl ? 2 : 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, k_tc_gemm_pair<BN>, ta, tb, to, a);
  return e != cudaSuccess ? e : cudaGetLastError();
}

template <int BN>
cudaError_t launch_tc_gemm_quad_bn(const TcGemm& g, int num_sms, cudaStream_t s) {
  using Cfg = Tc2Cfg<BN>;
  cudaError_t ea = cudaFuncSetAttribute(k_tc_gemm_quad<BN>,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kSmemBytes);
  if (ea != cudaSuccess) return ea;
  CUtensorMap ta, tbq, to;
  if (g.K % 8 != 0 || g.N % 4 != 0) return cudaErrorInvalidValue;
  if (g.out_bf16 && g.N % 8 != 0) return cudaErrorInvalidValue;
  if ((reinterpret_cast<uintptr_t>(g.out) & 15) != 0) return cudaErrorInvalidValue;
  if (!encode_kmajor_bf16(&ta, g.A, static_cast<uint64_t>(g.K),
                          static_cast<uint64_t>(g.E) * g.M, TC_BM) ||
      !encode_kmajor_bf16(&tbq, g.B, static_cast<uint64_t>(g.K),
                          static_cast<uint64_t>(g.E) * g.N, BN / 4) ||
      !encode_out_map(&to, g.out, g.E, g.M, g.N, g.out_bf16))
    return cudaErrorInvalidValue;
  TcArgs a;
  a.E = g.E;
  a.M = g.M;
  a.N = g.N;
  a.K = g.K;
  a.group_n = g.group_n > 0 ? g.group_n : (g.N + BN - 1) / BN;
  a.out = g.out;
  a.out_bf16 = g.out_bf16;
  a.alpha = g.alpha;
  a.flags = g.flags;
  a.stall = g.stall;
  a.sym_per_e = 0;  // clusters compute every tile (symmetric outputs run on pairs)
  const int Mt = (g.M + TC2_BM - 1) / TC2_BM, Nt = (g.N + BN - 1) / BN;
  const int64_t tiles = static_cast<int64_t>(g.E) * ((Mt + 1) / 2) * Nt;
  int clusters = num_sms / 4;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[2];
  pdl_attr(attr[1]);
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 4;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.blockDim = dim3(TC_THREADS, 1, 1);
  cfg.dynamicSmemBytes = Cfg::kSmemBytes;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cfg.gridDim = dim3(4 * clusters, 1, 1);
  int max_clusters = 0;
  if (cudaOccupancyMaxActiveClusters(&max_clusters, k_tc_gemm_quad<BN>, &cfg) != cudaSuccess ||
      max_clusters < 1) {
    cudaGetLastError();
    return launch_tc_gemm_pair_bn<BN>(g, num_sms, s);  // no 4-CTA cluster fits: pairs
  }
  if (max_clusters < clusters) clusters = max_clusters;
  if (tiles < clusters) clusters = static_cast<int>(tiles);
  cfg.gridDim = dim3(4 * clusters, 1, 1);
  cfg.numAttrs = g.pdl ? 2 : 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, k_tc_gemm_quad<BN>, ta, tbq, to, a);
  return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace

bool tc_gemm_supported(int device) { return tc_supported_impl(device); }

int tc_gemm_tile_n(int E, int M, int N, int num_sms, int pair) {
  if (pair) {
    // CTA pairs (256-row tiles over two SMs, 6-stage rings at both widths): 256-wide
    // tiles unless they take more waves x width than 224-wide ones.  Measured on
    // GB300: 4096 x 14336 886 vs 955 us, 28672 x 8192 2.11 vs 2.21 ms, 64 experts
    // 2048 x 7168 7.27 vs 7.69 ms; on 4096 x 4096, 224 wide (4 full waves) wins.
    const int pairs = num_sms / 2 > 0 ? num_sms / 2 : 1;
    const int64_t mt2 = (M + 255) / 256;
    auto pcost = [&](int bn) {
      const int64_t tiles = static_cast<int64_t>(E) * mt2 * ((N + bn - 1) / bn);
      return static_cast<double>((tiles + pairs - 1) / pairs) * bn;
    };
    return pcost(256) <= pcost(224) ? 256 : 224;
  }
  // 224-wide tiles by default: their 44 KiB stages give a 5-deep ring against 4 for
  // 256-wide ones, which measured faster on GB300 on every layer shape here (4096 x
  // 4096: 99 vs 111 us; 4096 x 14336: 1.00 vs 1.03 ms; 64 experts 2048 x 7168: 8.26
  // vs 8.58 ms), unless the wave count (waves x width) makes them clearly worse.
  // 128-wide tiles only when 256-wide ones leave many SMs idle and 128 balances far
  // better (on the 4096 x 4096 layer they lose: 140 us).
  const int64_t mt = (M + TC_BM - 1) / TC_BM;
  auto cost = [&](int bn) {
    const int64_t tiles = static_cast<int64_t>(E) * mt * ((N + bn - 1) / bn);
    return static_cast<double>((tiles + num_sms - 1) / num_sms) * bn;
  };
  const double b256 = wave_balance(static_cast<int64_t>(E) * mt * ((N + 255) / 256), num_sms);
  const double b128 = wave_balance(static_cast<int64_t>(E) * mt * ((N + 127) / 128), num_sms);
  if (b256 < 0.6 && b128 > b256 + 0.25) return 128;
  return cost(224) <= 1.1 * cost(256) ? 224 : 256;
}

namespace {

// Resident clusters of `csize` CTAs of `kernel` (its shared memory attribute set), 0 on error.
template <class Kern>
int resident_clusters(Kern kernel, int smem, int csize, int num_sms) {
  if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) !=
      cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = csize;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.blockDim = dim3(TC_THREADS, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cfg.gridDim = dim3(csize * (num_sms / csize), 1, 1);
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, kernel, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n < num_sms / csize ? n : num_sms / csize;
}

template <int BN>
int cluster_mode_bn(int E, int M, int N, int num_sms) {
  const int pairs = resident_clusters(k_tc_gemm_pair<BN>, Tc2Cfg<BN>::kSmemBytes, 2, num_sms);
  const int quads = resident_clusters(k_tc_gemm_quad<BN>, Tc2Cfg<BN>::kSmemBytes, 4, num_sms);
  if (pairs < 1 || quads < 1) return 3;
  const int64_t mt = (M + TC2_BM - 1) / TC2_BM, nt = (N + BN - 1) / BN;
  const int64_t pw = (static_cast<int64_t>(E) * mt * nt + pairs - 1) / pairs;
  const int64_t qw = (static_cast<int64_t>(E) * ((mt + 1) / 2) * nt + quads - 1) / quads;
  // Clusters read 23% less operand data per SM and ran each tile 5-8% faster on
  // GB300, where fewer 4-CTA clusters than 76 pairs are resident: 64 experts
  // 2048 x 7168, 200 waves against 189, 2.6% faster; 28672 x 8192, 50 against
  // 48, 0.5-0.9% faster; 4096 x 14336, 13 against 12, 3.6% slower; 4096 x 4096,
  // 5 against 4, 19% slower.  So clusters when they cost at most 6% more waves;
  // a contraction of a few waves keeps the pairs.
  if (pw < 4) return 3;
  return static_cast<double>(qw) <= 1.06 * static_cast<double>(pw) ? 2 : 3;
}

}  // namespace

int tc_gemm_cluster_mode(int E, int M, int N, int bn, int num_sms) {
  if (num_sms < 4) return 3;
  if (bn == 128) return cluster_mode_bn<128>(E, M, N, num_sms);
  if (bn == 224) return cluster_mode_bn<224>(E, M, N, num_sms);
  return cluster_mode_bn<256>(E, M, N, num_sms);
}

// Tile width of a symmetric output's upper triangle: 224 or 256, whichever costs fewer
// waves x width (4096 x 4096 on pairs: 136 tiles 256 wide, 2 waves, against 173 tiles
// 224 wide, 3 waves).
int sym_tile_n(int E, int M, int num_sms, int pair) {
  const int units = pair ? (num_sms / 2 > 0 ? num_sms / 2 : 1) : (num_sms > 0 ? num_sms : 1);
  const int bm = pair ? TC2_BM : TC_BM;
  auto cost = [&](int bn) {
    const int64_t tiles = static_cast<int64_t>(E) * upper_tiles(M, bm, bn);
    return static_cast<double>((tiles + units - 1) / units) * bn;
  };
  return cost(256) <= cost(224) ? 256 : 224;
}

cudaError_t launch_tc_gemm(const TcGemm& g, int num_sms, cudaStream_t s) {
  if (g.sym && g.M != g.N) return cudaErrorInvalidValue;
  const int bn = g.tile_n ? g.tile_n
                          : (g.sym ? sym_tile_n(g.E, g.M, num_sms, g.pair)
                                   : tc_gemm_tile_n(g.E, g.M, g.N, num_sms, g.pair));
  int mode = g.pair == 1 ? tc_gemm_cluster_mode(g.E, g.M, g.N, bn, num_sms) : g.pair;
  if (g.sym && mode == 2) mode = 3;  // the upper-triangle order runs on pairs
  if (mode == 2 && num_sms >= 4) {
    if (bn == 128) return launch_tc_gemm_quad_bn<128>(g, num_sms, s);
    if (bn == 224) return launch_tc_gemm_quad_bn<224>(g, num_sms, s);
    return launch_tc_gemm_quad_bn<256>(g, num_sms, s);
  }
  if (g.pair && num_sms >= 2) {
    if (bn == 128) return launch_tc_gemm_pair_bn<128>(g, num_sms, s);
    if (bn == 224) return launch_tc_gemm_pair_bn<224>(g, num_sms, s);
    return launch_tc_gemm_pair_bn<256>(g, num_sms, s);
  }
  if (bn == 128) return launch_tc_gemm_bn<128>(g, num_sms, s);
  if (bn == 224) return launch_tc_gemm_bn<224>(g, num_sms, s);
  return launch_tc_gemm_bn<256>(g, num_sms, s);
}

}  // namespace gsq
