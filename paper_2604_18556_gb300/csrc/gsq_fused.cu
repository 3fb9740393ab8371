// Fused optimisation step on the 5th-generation tensor cores (sm_103a): the loss
// contraction and everything that consumes its result, in one persistent kernel.
//
// For a tile of 128 weight columns c x 96 weight rows r of one expert:
//   contraction  A[c][r] = sum_j H[c][j] D_t[r][j]  (tcgen05.mma, bf16 operands, fp32
//                in TMEM).  H is symmetric, so A = (D_t H)^T and G = 2 A^T is the
//                gradient dL/dW^ of L = tr(D H D^T) (Eq. 1 with a linear layer).
//   epilogue     per weight (r, c) of the tile: step t's relaxation recomputed (Alg. 1),
//                the loss term 1/2 D G, the logit gradients (softmax Jacobian, App. B),
//                Lion on logits and momenta (§3.3), the group's scale gradient and its
//                Lion update, then the forward of step t + 1 (the next D): the same
//                arithmetic as the separate backward kernel.
// G never reaches HBM, and the MMAs of the next tiles run while this tile's
// elementwise work does.
//
// Warps (16, one CTA per SM, at most 4 per SM sub-partition: 128 registers a thread):
//   warp 0      TMA producer: 128 x 64 tiles of H and 96 x 64 tiles of D_t per stage,
//               128-byte swizzle, 4-stage ring;
//   warp 1      TMEM allocator and MMA issuer (M = 128, N = 96, K = 16); the accumulator
//               is double-buffered in TMEM;
//   warps 2-15  epilogue.  Per tile, 12 of them, three per TMEM lane quarter (warp mod 4),
//               each copy one 32 x 32 block of the accumulator into a shared 96 x 128
//               fp32 tile (double-buffered by tile parity, so warps done with a tile go
//               on to the next; one bounded mbarrier round per tile), then the 14
//               warps take whole 128-column rows of it from a shared counter: a thread owns
//               a quad of 4 consecutive weights (float4 state loads, 512 contiguous
//               bytes per plane per row), exactly as in the separate backward kernel,
//               and a scale group (at most 128 columns) lies in one warp, so its sum is
//               a warp shuffle.  The producer and MMA warps wait with the hardware's
//               suspending mbarrier test; the epilogue warps back off with short sleeps.
//               The loss is summed per row (a fixed shuffle tree) into
//               per-row accumulators, so the result does not depend on which warp took
//               which row.
// D_{t+1} is written to the other D buffer: tiles still being contracted read D_t.
// Every wait is bounded (kWaitLimitNs of %globaltimer); on expiry the CTA raises its
// abort flag, unwinds (the producer first waits, bounded, for its copies in flight),
// frees its TMEM and records an error code in the workspace flags.
#include <cuda.h>
#include <cuda_bf16.h>
#include <stddef.h>

#include "gsq_internal.h"
#include "gsq_relax.cuh"
#include "gsq_tc.cuh"

namespace gsq {
namespace {

constexpr int FZ_BM = 128;                   // weight columns per tile (TMEM lanes)
constexpr int FZ_BN = 96;                    // weight rows per tile (TMEM columns)
constexpr int FZ_BK = 64;                    // contraction per stage (one 128-byte row)
constexpr int FZ_BLOCKS = FZ_BN / 32;        // 32-row accumulator blocks per lane quarter
constexpr int FZ_DUMPERS = 4 * FZ_BLOCKS;    // warps copying the accumulator to shared memory
constexpr int FZ_EPI_WARPS = 14;
constexpr int FZ_THREADS = 32 * (2 + FZ_EPI_WARPS);
constexpr int FZ_A_BYTES = FZ_BM * FZ_BK * 2;
constexpr int FZ_STAGE_BYTES = (FZ_BM + FZ_BN) * FZ_BK * 2;
constexpr int FZ_STAGES = 4;
constexpr int FZ_ACC_STRIDE = 128;           // TMEM column offset of the second accumulator
constexpr int FZ_TMEM_COLS = 256;
// kind::f16 instruction descriptor: D fp32, A and B bf16, both K-major, N >> 3, M >> 4.
constexpr uint32_t FZ_IDESC = (1u << 4) | (1u << 7) | (1u << 10) |
                              (static_cast<uint32_t>(FZ_BN >> 3) << 17) |
                              (static_cast<uint32_t>(FZ_BM >> 4) << 24);
static_assert(FZ_BN <= FZ_ACC_STRIDE && 2 * FZ_ACC_STRIDE == FZ_TMEM_COLS, "TMEM layout");
static_assert(FZ_STAGE_BYTES % 1024 == 0 && FZ_A_BYTES % 1024 == 0, "128-byte swizzle atoms");
static_assert(FZ_THREADS == 512, "16 warps: at most 4 per SM sub-partition (128 registers)");
static_assert(FZ_DUMPERS <= FZ_EPI_WARPS, "a dumping warp per accumulator block");

// Shared control block after the ring (1024-byte aligned; the float4-read tile first).
struct FzCtl {
  alignas(16) float G[2][FZ_BN][FZ_BM];  // G of the tile, by tile parity
  uint64_t full[FZ_STAGES], empty[FZ_STAGES];
  uint64_t tfull[2], tempty[2];          // accumulator published / free
  uint64_t ready[2], consumed[2];        // shared G tile written / read by every warp
  double row_loss[2][FZ_BN];             // loss of row r summed over this CTA's tiles
  int rows_next[2];                      // row counters, by tile parity
  float sgrid[kMaxLevels];
  uint32_t tmem_slot;
  int abort;
  int is_last;
};
constexpr int FZ_SMEM_BYTES = FZ_STAGES * FZ_STAGE_BYTES + 1024 + static_cast<int>(sizeof(FzCtl));
static_assert(FZ_SMEM_BYTES <= 232448, "shared memory per CTA");
static_assert((FZ_STAGES * FZ_STAGE_BYTES) % 1024 == 0 && offsetof(FzCtl, G) == 0 &&
                  offsetof(FzCtl, full) % 8 == 0,
              "control block alignment");

struct FusedArgs {
  EwParams P;     // state, noise, step t and t + 1, Lion (P.D unused: D_t is read by TMA)
  void* D_next;   // bf16 [n]: receives D_{t+1} when P.lookahead
  float* G_out;   // nullable: also store G (fp32 [n])
  int E, R, C;
  int group_n;    // tile order: groups of row tiles (tile_coords)
};

// Sixteen consecutive accumulator columns (weight rows) of this thread's TMEM lane.
__device__ __forceinline__ void tmem_ld16x(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, "
      "%12, %13, %14, %15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// Bounded wait taken by lane 0 for the whole warp: every lane leaves with the same
// answer, so the warp-collective instructions after it stay converged.  The
// shuffle also orders lane 0's acquire before the other lanes' later reads.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                          uint32_t max_sleep_ns) {
  int ok = 1;
  if ((threadIdx.x & 31) == 0)
    ok = mbar_wait_backoff(bar, parity, abort_flag, max_sleep_ns) ? 1 : 0;
  return __shfl_sync(0xffffffffu, ok, 0) != 0;
}

// Back-off ceiling (ns) of the epilogue warps' waits.
constexpr uint32_t kSleepEpilogue = 256;

template <class Rx, bool kShift>
__global__ void __launch_bounds__(FZ_THREADS, 1)
    k_step_fused(const __grid_constant__ CUtensorMap tmH, const __grid_constant__ CUtensorMap tmD,
                 const FusedArgs a) {
  constexpr int K = Rx::L;
  const EwParams& P = a.P;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  FzCtl* ctl = reinterpret_cast<FzCtl*>(smem + FZ_STAGES * FZ_STAGE_BYTES);
  volatile int* abort_flag = &ctl->abort;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < FZ_STAGES; ++s) {
      mbar_init(ctl->full + s, 1);
      mbar_init(ctl->empty + s, 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(ctl->tfull + b, 1);
      mbar_init(ctl->tempty + b, FZ_DUMPERS);
      ctl->rows_next[b] = 0;
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(ctl->ready + b, FZ_DUMPERS);
      mbar_init(ctl->consumed + b, FZ_EPI_WARPS);
      for (int r = 0; r < FZ_BN; ++r) ctl->row_loss[b][r] = 0.0;
    }
    ctl->abort = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmH)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmD)) : "memory");
  }
  if (threadIdx.x < kMaxLevels) ctl->sgrid[threadIdx.x] = P.grid[threadIdx.x];
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(&ctl->tmem_slot)),
                 "r"(FZ_TMEM_COLS));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = ctl->tmem_slot;

  const int Mt = (a.C + FZ_BM - 1) / FZ_BM;  // column tiles (rows of H)
  const int Nt = (a.R + FZ_BN - 1) / FZ_BN;  // row tiles (rows of D)
  const int KB = (a.C + FZ_BK - 1) / FZ_BK;
  const int tiles = a.E * Mt * Nt;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      int stage = 0;
      uint32_t phase = 0;
      uint32_t issued_phase[FZ_STAGES];
      bool issued[FZ_STAGES];
      for (int s = 0; s < FZ_STAGES; ++s) issued[s] = false;
      bool ok = true;
      for (int tile = blockIdx.x; ok && tile < tiles; tile += gridDim.x) {
        int e, m, n;
        tile_coords(tile, Mt, Nt, a.group_n, e, m, n);
        const int hrow = e * a.C + m * FZ_BM;
        const int drow = e * a.R + n * FZ_BN;
        for (int kb = 0; kb < KB; ++kb) {
          if (!mbar_wait(ctl->empty + stage, phase ^ 1u, abort_flag)) {
            ok = false;
            break;
          }
          uint8_t* sa = smem + stage * FZ_STAGE_BYTES;
          mbar_expect_tx(ctl->full + stage, FZ_STAGE_BYTES);
          tma_load_2d(sa, &tmH, ctl->full + stage, kb * FZ_BK, hrow);
          tma_load_2d(sa + FZ_A_BYTES, &tmD, ctl->full + stage, kb * FZ_BK, drow);
          issued[stage] = true;
          issued_phase[stage] = phase;
          if (++stage == FZ_STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok) {
        // abort: wait (bounded, ignoring the abort flag) for our own copies in flight
        for (int s = 0; s < FZ_STAGES; ++s)
          if (issued[s]) mbar_wait(ctl->full + s, issued_phase[s], abort_flag, false);
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
        if (!mbar_wait(ctl->tempty + acc, acc_phase ^ 1u, abort_flag)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * FZ_ACC_STRIDE);
        for (int kb = 0; kb < KB; ++kb) {
          if (!mbar_wait(ctl->full + stage, phase, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + stage * FZ_STAGE_BYTES);
          const uint64_t da = sw128_desc(sa);
          const uint64_t db = sw128_desc(sa + FZ_A_BYTES);
#pragma unroll
          for (int k = 0; k < FZ_BK / 16; ++k)
            umma_bf16(d_tmem, da + 2 * k, db + 2 * k, FZ_IDESC, (kb | k) != 0 ? 1u : 0u);
          umma_commit(ctl->empty + stage);
          if (++stage == FZ_STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
        if (!ok) break;
        umma_commit(ctl->tfull + acc);
        if (++acc == 2) {
          acc = 0;
          acc_phase ^= 1u;
        }
      }
    }
  } else {
    // ---------------- epilogue: backward + Lion + look-ahead forward ----------------
    const int quarter = warp & 3;  // the TMEM lane quarter this warp may read
    // its 32-row block of the accumulator, if any: the warps of each quarter from the first
    // epilogue warp of that quarter (warps 4, 5, 2, 3) take blocks 0, 1, 2 in turn
    const int first = quarter < 2 ? quarter + 4 : quarter;
    const int blk = (warp - first) >> 2;
    const bool dumper = blk < FZ_BLOCKS;
    float q[kMaxLevels];
#pragma unroll
    for (int k = 0; k < kMaxLevels; ++k) q[k] = P.grid[k];
    const int seg = P.group >> 2;  // lanes per scale group (a group lies in one row)
    const bool frozen = P.scales_frozen != 0;
    // Tile lj's accumulator goes to shared buffer lj & 1.  Each copying warp copies
    // tile li + 1 before it processes tile li, so a warp can run a tile ahead of the
    // slowest one.
    const int my_tiles = (tiles - static_cast<int>(blockIdx.x) + static_cast<int>(gridDim.x) - 1) /
                         static_cast<int>(gridDim.x);
    auto dump = [&](int lj) -> bool {
      const int b = lj & 1;
      const uint32_t ph = (lj >> 1) & 1u;
      if (!warp_wait(ctl->tfull + b, ph, abort_flag, kSleepEpilogue)) return false;
      tc_fence_after();
      // every warp has finished tile lj - 2, the last user of this buffer
      if (lj >= 2 && !warp_wait(ctl->consumed + b, ph ^ 1u, abort_flag, kSleepEpilogue)) return false;
      if (warp == 2 && lane == 0) ctl->rows_next[b] = 0;  // tile lj - 2's counter: all done
      float (*Gt)[FZ_BM] = ctl->G[b];
      const uint32_t taddr = tmem_base + static_cast<uint32_t>(b * FZ_ACC_STRIDE + 32 * blk) +
                             (static_cast<uint32_t>(quarter * 32) << 16);
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        float v[16];
        tmem_ld16x(taddr + 16 * h, v);
#pragma unroll
        for (int i = 0; i < 16; ++i) Gt[32 * blk + 16 * h + i][32 * quarter + lane] = 2.0f * v[i];
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(ctl->tempty + b);
        mbar_arrive(ctl->ready + b);
      }
      return true;
    };
    bool ok = !(dumper && my_tiles > 0) || dump(0);
    for (int li = 0; ok && li < my_tiles; ++li) {
      if (dumper && li + 1 < my_tiles && !dump(li + 1)) break;
      const int tile = static_cast<int>(blockIdx.x) + li * static_cast<int>(gridDim.x);
      const int b = li & 1;
      float (*Gt)[FZ_BM] = ctl->G[b];
      if (!warp_wait(ctl->ready + b, (li >> 1) & 1u, abort_flag, kSleepEpilogue)) break;
      int e, m, n;
      tile_coords(tile, Mt, Nt, a.group_n, e, m, n);
      const int c = m * FZ_BM + 4 * lane;
      const bool col_ok = c < a.C;  // C % 8 == 0: a quad is wholly inside or outside
#pragma unroll 1
      while (true) {
        int rl = 0;
        if (lane == 0) rl = atomicAdd(&ctl->rows_next[b], 1);
        rl = __shfl_sync(0xffffffffu, rl, 0);
        if (rl >= FZ_BN) break;
        const int r = n * FZ_BN + rl;
        const bool active = col_ok && r < a.R;
        const int64_t qi = ((static_cast<int64_t>(e) * a.R + r) * a.C + c) >> 2;
        const int64_t qc = active ? qi : 0;
        float l[K][4], m4[K][4];
        float w[4];
#pragma unroll
        for (int k = 0; k < K; ++k) {
          const float4 v = __ldcs(reinterpret_cast<const float4*>(P.logits + k * P.n) + qc);
          l[k][0] = v.x; l[k][1] = v.y; l[k][2] = v.z; l[k][3] = v.w;
          const float4 u = __ldcs(reinterpret_cast<const float4*>(P.m_logits + k * P.n) + qc);
          m4[k][0] = u.x; m4[k][1] = u.y; m4[k][2] = u.z; m4[k][3] = u.w;
        }
        load_w4(P.W, qc, P.w_bf16, w);
        const int64_t gidx = (qc * 4) >> P.log2_group;
        float s = __ldg(P.scales + gidx);
        float ms = frozen ? 0.0f : __ldg(P.m_scales + gidx);
        const uint32_t j4 = kShift ? load_j0(P, qc) : 0u;
        float4 gv = *reinterpret_cast<const float4*>(&Gt[rl][4 * lane]);
        if (!active) gv = make_float4(0.f, 0.f, 0.f, 0.f);
        const float2 Gq[2] = {make_float2(gv.x, gv.y), make_float2(gv.z, gv.w)};
        float2 ds2 = f2(0.0f), loss2 = f2(0.0f);
#pragma unroll
        for (int pr = 0; pr < 2; ++pr) {
          float2 l2[K], h[K];
#pragma unroll
          for (int k = 0; k < K; ++k) l2[k] = make_float2(l[k][2 * pr], l[k][2 * pr + 1]);
          Rx rx(q, ctl->sgrid, P.nlev, (j4 >> (16 * pr)) & 0xFFu, (j4 >> (16 * pr + 8)) & 0xFFu);
          Rx::noise(P.keys, P.t, static_cast<uint64_t>(qc) * 4 + 2 * pr, P.noise, h);
          const float2 wt = rx.relax(l2, h, P.kappa_log2, P.inv_tau);
          const float2 dd = fma2(f2(s), wt, make_float2(-w[2 * pr], -w[2 * pr + 1]));
          const float2 dj = make_float2(round_d(dd.x, 1), round_d(dd.y, 1));
          loss2 = fma2(mul2(f2(0.5f), dj), Gq[pr], loss2);
          ds2 = fma2(Gq[pr], wt, ds2);
          const float2 A = mul2(f2(P.kappa_over_tau * s), Gq[pr]);
#pragma unroll
          for (int k = 0; k < K; ++k) {
            // dL/dl_k = (kappa/tau) G s dw~/dl_k, then Lion with decoupled decay
            const float2 dl = mul2(A, rx.dsoft(k));
            const float2 mo = make_float2(m4[k][2 * pr], m4[k][2 * pr + 1]);
            const float2 cm = fma2(f2(P.b1), mo, mul2(f2(1.0f - P.b1), dl));
            const float2 ln = add2(fma2(f2(-P.lrwd_l), l2[k], l2[k]),
                                   make_float2(-lr_sign(P.lr_l, cm.x), -lr_sign(P.lr_l, cm.y)));
            const float2 mn = fma2(f2(P.b2), mo, mul2(f2(1.0f - P.b2), dl));
            l[k][2 * pr] = ln.x; l[k][2 * pr + 1] = ln.y;
            m4[k][2 * pr] = mn.x; m4[k][2 * pr + 1] = mn.y;
          }
        }
        if (active) {
#pragma unroll
          for (int k = 0; k < K; ++k) {
            __stcs(reinterpret_cast<float4*>(P.logits + k * P.n) + qi,
                   make_float4(l[k][0], l[k][1], l[k][2], l[k][3]));
            __stcs(reinterpret_cast<float4*>(P.m_logits + k * P.n) + qi,
                   make_float4(m4[k][0], m4[k][1], m4[k][2], m4[k][3]));
          }
          if (a.G_out) reinterpret_cast<float4*>(a.G_out)[qi] = gv;
        }
        // the row's loss: a fixed fp32 shuffle tree, added to the row's fp64 accumulator
        float lr = loss2.x + loss2.y;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) lr += __shfl_xor_sync(0xffffffffu, lr, off);
        if (lane == 0) ctl->row_loss[b][rl] += static_cast<double>(lr);
        if (!frozen) {
          // dL/ds_g = sum over the group of G w~: seg lanes of this warp
          const float ds = group_sum(ds2.x + ds2.y, seg);
          const float cs = fmaf(P.b1, ms, (1.0f - P.b1) * ds);
          s = fmaf(-P.lrwd_s, s, s) - lr_sign(P.lr_s, cs);
          ms = fmaf(P.b2, ms, (1.0f - P.b2) * ds);
          if (active && (lane & (seg - 1)) == 0) {
            P.scales[gidx] = s;
            P.m_scales[gidx] = ms;
          }
        }
        if (P.lookahead && active) {
          // forward of step t + 1 from the updated logits and scale (Alg. 1)
          float d[4];
#pragma unroll
          for (int pr = 0; pr < 2; ++pr) {
            float2 l2[K], h[K];
#pragma unroll
            for (int k = 0; k < K; ++k) l2[k] = make_float2(l[k][2 * pr], l[k][2 * pr + 1]);
            const Rx rx(q, ctl->sgrid, P.nlev, (j4 >> (16 * pr)) & 0xFFu, (j4 >> (16 * pr + 8)) & 0xFFu);
            Rx::noise(P.keys, P.t_next, static_cast<uint64_t>(qi) * 4 + 2 * pr, P.noise, h);
            const float2 wt = rx.value(l2, h, P.kappa_log2_next, P.inv_tau_next);
            const float2 dd = fma2(f2(s), wt, make_float2(-w[2 * pr], -w[2 * pr + 1]));
            d[2 * pr] = dd.x;
            d[2 * pr + 1] = dd.y;
          }
          store_d4(a.D_next, qi, 1, d);
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(ctl->consumed + b);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();  // lane 0 ran the MMA loop: reconverge for the aligned dealloc
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem_base),
                 "r"(FZ_TMEM_COLS));
  }
  // deterministic loss: per-CTA partials summed in CTA order by the last CTA to finish
  if (threadIdx.x == 0) {
    double s = 0.0;
    for (int b = 0; b < 2; ++b)
      for (int r = 0; r < FZ_BN; ++r) s += ctl->row_loss[b][r];
    P.loss_partials[blockIdx.x] = s;
    __threadfence();
    const unsigned int prev = atomicAdd(&P.flags->blocks_done, 1u);
    ctl->is_last = prev == gridDim.x - 1;
    if (ctl->is_last) {
      __threadfence();
      double tot = 0.0;
      for (unsigned int b = 0; b < gridDim.x; ++b) tot += __ldcg(P.loss_partials + b);
      if (P.loss_out) *P.loss_out = static_cast<float>(tot);
      P.flags->blocks_done = 0u;
    }
    if (*abort_flag) atomicExch(&P.flags->error, 0x7C02u);
  }
}

template <class Rx, bool kShift>
cudaError_t launch_fused_impl(const CUtensorMap& tmH, const CUtensorMap& tmD, const FusedArgs& a,
                              int grid, cudaStream_t s) {
  // set on every launch: the attribute belongs to the current device
  const cudaError_t e = cudaFuncSetAttribute(
      k_step_fused<Rx, kShift>, cudaFuncAttributeMaxDynamicSharedMemorySize, FZ_SMEM_BYTES);
  if (e != cudaSuccess) return e;
  k_step_fused<Rx, kShift><<<grid, FZ_THREADS, FZ_SMEM_BYTES, s>>>(tmH, tmD, a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_step_fused(const FusedStep& f, int num_sms, cudaStream_t s) {
  if (f.C % 8 != 0 || f.E < 1 || f.R < 1) return cudaErrorInvalidValue;  // 16-byte TMA rows
  CUtensorMap tmH, tmD;
  if (!encode_kmajor_bf16(&tmH, f.H, static_cast<uint64_t>(f.C),
                          static_cast<uint64_t>(f.E) * f.C, FZ_BM) ||
      !encode_kmajor_bf16(&tmD, f.D_t, static_cast<uint64_t>(f.C),
                          static_cast<uint64_t>(f.E) * f.R, FZ_BN))
    return cudaErrorInvalidValue;
  FusedArgs a;
  a.P = f.P;
  a.D_next = f.D_next;
  a.G_out = f.G_out;
  a.E = f.E;
  a.R = f.R;
  a.C = f.C;
  const int Mt = (f.C + FZ_BM - 1) / FZ_BM, Nt = (f.R + FZ_BN - 1) / FZ_BN;
  a.group_n = f.group_n > 0 ? f.group_n : Nt;
  const int64_t tiles = static_cast<int64_t>(f.E) * Mt * Nt;
  const int grid = static_cast<int>(tiles < num_sms ? tiles : num_sms);
  cudaError_t err = cudaSuccess;
  const cudaError_t e = with_relax(f.P.K, f.P.mode, [&](auto rx, auto sh) {
    using Rx = typename decltype(rx)::type;
    err = launch_fused_impl<Rx, decltype(sh)::value>(tmH, tmD, a, grid, s);
  });
  return e != cudaSuccess ? e : err;
}

}  // namespace gsq
