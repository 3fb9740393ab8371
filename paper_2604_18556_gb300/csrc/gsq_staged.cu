// The fused backward with its input streams staged through shared memory by
// bulk asynchronous copies (k_backward_staged), for non-exporting steps: the
// kernel, its staging plans and its launch.
#include <cuda_bf16.h>

#include <cstdlib>
#include <type_traits>

#include "gsq_backward.cuh"
#include "gsq_internal.h"
#include "gsq_tc.cuh"

namespace gsq {
namespace {

// ---------------------------------------------------------------------------
// TMA-staged fused backward (non-export, non-accumulating steps): the per-quad
// body of k_backward, with the streams a block reads (logits, their momenta,
// G, W, scales, scale momenta, j0) brought into shared memory by bulk
// asynchronous copies (cp.async.bulk, completion counted on an mbarrier) a tile
// ahead, so the warps read them with shared-memory loads instead of stalling
// on HBM.  A tile is 256 quads (1,024 weights, one quad per thread); tiles go
// to blocks round-robin (tile = blockIdx.x + j * gridDim.x) through two stages.
// The last warp to finish reading a stage (a shared counter) issues the copies
// of the block's tile two ahead into it, so no warp waits for another.  A
// partial last tile is read with direct loads by the block whose turn it is.
// The plan decides which streams besides the logits are staged (plan 3, the
// default up to 4 logits, loads the logit momenta directly: they arrive while
// the noise is drawn).  Stores stay direct.
// Every wait is bounded (2 s of %globaltimer); on expiry the block records an
// error code, waits (bounded) for its own copies in flight and returns.
// ---------------------------------------------------------------------------
constexpr int kTileQ = kEwThreads;                 // quads per tile
constexpr int64_t kTileW = 4 * kTileQ;             // weights per tile
constexpr uint32_t kPlaneBytes = 4u * kTileW;      // one fp32 plane of a tile

// A staging plan: blocks per SM the registers are budgeted for, and which of the
// per-weight streams besides the logits go through shared memory (logit
// momenta; G and W).  Streams not staged are loaded directly at the top of the
// iteration.  Two stages of every resident block must fit in shared memory.
template <int kOcc_, bool kStageM_, bool kStageGW_>
struct StagePlan {
  static constexpr int kOcc = kOcc_;
  static constexpr bool kStageM = kStageM_;
  static constexpr bool kStageGW = kStageGW_;
};

__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// Copies of tile `tile` into stage `st`; the byte count the mbarrier expects
// is S.tx (the sum of the copies below).
template <int L, bool kShift, bool kStageM, bool kStageGW>
__device__ __forceinline__ void stage_issue(const EwParams& P, const BwdStage& S, unsigned char* st,
                                            uint64_t* bar, int64_t tile) {
  const int64_t w0 = tile * kTileW;
  mbar_expect_tx(bar, S.tx);
#pragma unroll
  for (int k = 0; k < L; ++k) bulk_g2s(st + S.l + k * kPlaneBytes, P.logits + k * P.n + w0, kPlaneBytes, bar);
  if (kStageM) {
#pragma unroll
    for (int k = 0; k < L; ++k)
      bulk_g2s(st + S.m + k * kPlaneBytes, P.m_logits + k * P.n + w0, kPlaneBytes, bar);
  }
  if (kStageGW) {
    bulk_g2s(st + S.g, P.G + w0, kPlaneBytes, bar);
    const int wb = P.w_bf16 ? 2 : 4;
    bulk_g2s(st + S.w, static_cast<const unsigned char*>(P.W) + w0 * wb,
             static_cast<uint32_t>(kTileW * wb), bar);
  }
  const uint32_t sb = kPlaneBytes >> P.log2_group;  // one fp32 per scale group
  bulk_g2s(st + S.s, P.scales + (w0 >> P.log2_group), sb, bar);
  if (!P.scales_frozen) bulk_g2s(st + S.ms, P.m_scales + (w0 >> P.log2_group), sb, bar);
  if (kShift) bulk_g2s(st + S.j, P.j0 + w0, static_cast<uint32_t>(kTileW), bar);
}

template <class Rx, bool kShift, class Plan>
__global__ void __launch_bounds__(kEwThreads, Plan::kOcc)
    k_backward_staged(const EwParams P, const BwdStage S) {
  constexpr int K = Rx::L;
  constexpr bool kStageM = Plan::kStageM;
  constexpr bool kStageGW = Plan::kStageGW;
  constexpr unsigned int kWarps = kEwThreads / 32;
  extern __shared__ __align__(128) unsigned char stage_mem[];
  __shared__ __align__(8) uint64_t full[2];
  __shared__ unsigned int done[2], issued[2];
  __shared__ int abort_flag;
  __shared__ float sgrid[kMaxLevels];
  grid_dep_wait();
  grid_dep_launch();
  float q[kMaxLevels];
  load_grid(P, q);
  const int tid = threadIdx.x, lane = tid & 31;
  const int seg = P.group >> 2;  // lanes per scale group
  const int64_t ntiles = P.nq / kTileQ;  // full tiles
  const int64_t first = blockIdx.x, stride = gridDim.x;
  volatile int* abort_v = &abort_flag;
  if (tid == 0) {
    mbar_init(&full[0], 1);
    mbar_init(&full[1], 1);
    done[0] = done[1] = 0u;
    issued[0] = issued[1] = 0u;
    abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (kShift && tid < kMaxLevels) sgrid[tid] = P.grid[tid];
  __syncthreads();
  if (tid == 0) {
#pragma unroll
    for (int b = 0; b < 2; ++b) {
      if (first + b * stride < ntiles && !(P.stall && b == 1)) {
        stage_issue<K, kShift, kStageM, kStageGW>(P, S, stage_mem + b * S.bytes, &full[b], first + b * stride);
        issued[b] = 1u;
      }
    }
  }
  float2 loss2 = f2(0.0f);
  int64_t j = 0;
  for (int64_t tile = first; tile < ntiles; tile += stride, ++j) {
    const int b = static_cast<int>(j & 1);
    const uint32_t parity = static_cast<uint32_t>((j >> 1) & 1);
    const bool ok = __all_sync(0xffffffffu, mbar_wait(&full[b], parity, abort_v) ? 1 : 0);
    if (!ok) break;
    const unsigned char* st = stage_mem + b * S.bytes;
    const int64_t qi = tile * kTileQ + tid;
    float l[K][4], m[K][4], w[4];
#pragma unroll
    for (int k = 0; k < K; ++k) {
      const float4 v = reinterpret_cast<const float4*>(st + S.l + k * kPlaneBytes)[tid];
      l[k][0] = v.x; l[k][1] = v.y; l[k][2] = v.z; l[k][3] = v.w;
    }
#pragma unroll
    for (int k = 0; k < K; ++k) {
      const float4 v = kStageM ? reinterpret_cast<const float4*>(st + S.m + k * kPlaneBytes)[tid]
                               : __ldcs(reinterpret_cast<const float4*>(P.m_logits + k * P.n) + qi);
      m[k][0] = v.x; m[k][1] = v.y; m[k][2] = v.z; m[k][3] = v.w;
    }
    float4 gv;
    if (!kStageGW) {
      gv = __ldcs(reinterpret_cast<const float4*>(P.G) + qi);
      load_w4(P.W, qi, P.w_bf16, w);
    } else {
      gv = reinterpret_cast<const float4*>(st + S.g)[tid];
      if (P.w_bf16) {
        const uint2 raw = reinterpret_cast<const uint2*>(st + S.w)[tid];
        const float2 fa = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&raw.x));
        const float2 fb = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&raw.y));
        w[0] = fa.x; w[1] = fa.y; w[2] = fb.x; w[3] = fb.y;
      } else {
        const float4 v = reinterpret_cast<const float4*>(st + S.w)[tid];
        w[0] = v.x; w[1] = v.y; w[2] = v.z; w[3] = v.w;
      }
    }
    const int gl = (tid * 4) >> P.log2_group;  // scale group within the tile
    const float s = reinterpret_cast<const float*>(st + S.s)[gl];
    const float ms = P.scales_frozen ? 0.0f : reinterpret_cast<const float*>(st + S.ms)[gl];
    const uint32_t j4 = kShift ? reinterpret_cast<const uint32_t*>(st + S.j)[tid] : 0u;
    // Release the stage: the warp that completes the count refills it with this
    // block's tile two ahead (generic reads ordered before the async-proxy writes).
    __syncwarp();
    if (lane == 0) {
      __threadfence_block();
      const unsigned int prev = atomicAdd(&done[b], 1u);
      if ((prev + 1u) % kWarps == 0u) {
        const int64_t nxt = tile + 2 * stride;
        if (nxt < ntiles) {
          __threadfence_block();
          asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
          stage_issue<K, kShift, kStageM, kStageGW>(P, S, stage_mem + b * S.bytes, &full[b], nxt);
          issued[b] += 1u;
        }
      }
    }
    bwd_quad<Rx, false, kShift, false>(P, q, sgrid, lane, seg, qi, true, l, m, gv, w, s, ms, j4,
                                       loss2);
  }
  __syncthreads();
  if (*abort_v) {
    // wait (bounded, ignoring the abort flag) for the copies still in flight into
    // this block's stages before the block leaves
    if (tid == 0) {
#pragma unroll
      for (int b = 0; b < 2; ++b)
        if (issued[b]) mbar_wait(&full[b], (issued[b] - 1u) & 1u, abort_v, false);
    }
  } else if (ntiles * kTileQ < P.nq && first == ntiles % stride) {
    // the partial last tile, with direct loads
    const int64_t qi = ntiles * kTileQ + tid;
    const bool active = qi < P.nq;
    float l[K][4], m[K][4], w[4];
    float4 gv;
    float s, ms;
    uint32_t j4;
    bwd_load_global<K, false, kShift>(P, qi, active, l, m, gv, w, s, ms, j4);
    bwd_quad<Rx, false, kShift, false>(P, q, sgrid, lane, seg, qi, active, l, m, gv, w, s, ms, j4,
                                       loss2);
  }
  reduce_loss(loss2.x + loss2.y, P);
  if (tid == 0 && *abort_v) atomicExch(&P.flags->error, 0x7C03u);
}

}  // namespace

namespace {

BwdStage stage_layout(int L, bool stage_m, bool stage_gw, int w_bf16, int log2_group,
                      int scales_frozen, int shift) {
  auto up = [](uint32_t x) { return (x + 127u) & ~127u; };
  BwdStage S{};
  const uint32_t sb = kPlaneBytes >> log2_group;
  const uint32_t wbytes = static_cast<uint32_t>(kTileW) * (w_bf16 ? 2u : 4u);
  uint32_t off = 0, tx = 0;
  S.l = off; off += L * kPlaneBytes; tx += L * kPlaneBytes;
  S.m = off;
  if (stage_m) { off += L * kPlaneBytes; tx += L * kPlaneBytes; }
  S.g = off;
  if (stage_gw) { off += kPlaneBytes; tx += kPlaneBytes; }
  S.w = off;
  if (stage_gw) { off += up(wbytes); tx += wbytes; }
  S.s = off; off += up(sb); tx += sb;
  S.ms = off;
  if (!scales_frozen) { off += up(sb); tx += sb; }
  S.j = off;
  if (shift) { off += static_cast<uint32_t>(kTileW); tx += static_cast<uint32_t>(kTileW); }
  S.bytes = (off + 1023u) & ~1023u;
  S.tx = tx;
  return S;
}

// Staging plans (the plan id is kept by the layer), measured on GB300 against
// each other and against the direct-load kernel:
//   1: 2 blocks/SM, every stream staged (tuning alternative);
//   3: 3 blocks/SM (80 registers, up to 4 logits per weight), logits, G, W and
//      scales staged, logit momenta loaded directly: fastest up to 4 logits;
//   5: 2 blocks/SM, as 3 with the register budget of 2 blocks: fastest from 6
//      logits up.
// With 5 logits (local shift) the direct-load kernel was faster than every
// plan, so none is chosen there.
using Plan1 = StagePlan<2, true, true>;
using Plan3 = StagePlan<3, false, true>;
using Plan5 = StagePlan<2, false, true>;

int default_plan(int L) { return L <= 4 ? 3 : (L == 5 ? 0 : 5); }

template <int L, class F>
void with_plan(int plan, F&& f) {
  switch (plan) {
    case 1: f(Plan1{}); break;
    case 3: if constexpr (L <= 4) f(Plan3{}); break;
    case 5: f(Plan5{}); break;
    default: break;
  }
}

template <class Rx, bool kShift, class Plan>
int staged_grid_for(const BwdStage& S, int num_sms) {
  auto* fn = k_backward_staged<Rx, kShift, Plan>;
  const int dyn = 2 * static_cast<int>(S.bytes);
  if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, dyn) != cudaSuccess ||
      cudaFuncSetAttribute(fn, cudaFuncAttributePreferredSharedMemoryCarveout, 100) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, reinterpret_cast<const void*>(fn),
                                                    kEwThreads, dyn) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  // only where the blocks the plan budgets its registers for are resident
  return per_sm >= Plan::kOcc ? per_sm * num_sms : 0;
}

}  // namespace

int ew_staged_grid(int K, int mode, int w_bf16, int log2_group, int scales_frozen, int num_sms,
                   int* plan_out) {
  *plan_out = 0;
  if (log2_group < 2 || log2_group > 7) return 0;
  int g = 0;
  with_relax(K, mode, [&](auto rx, auto sh) {
    using Rx = typename decltype(rx)::type;
    constexpr bool SH = decltype(sh)::value;
    int plan = default_plan(Rx::L);
    if (const char* e = std::getenv("GSQ_STAGED_PLAN")) {  // tuning override: 1, 3 or 5
      const int v = std::atoi(e);
      if (v == 1 || v == 3 || v == 5) plan = v;
    }
    with_plan<Rx::L>(plan, [&](auto pl) {
      using Plan = decltype(pl);
      const BwdStage S = stage_layout(Rx::L, Plan::kStageM, Plan::kStageGW, w_bf16, log2_group,
                                      scales_frozen, SH ? 1 : 0);
      g = staged_grid_for<Rx, SH, Plan>(S, num_sms);
      if (g > 0) *plan_out = plan;
    });
  });
  return g;
}

cudaError_t launch_backward_staged(const EwParams& p, int grid, int plan, cudaStream_t s,
                                   bool pdl) {
  if (p.grad_logits || p.grad_scales || p.acc_in_l || p.acc_in_s) return cudaErrorInvalidValue;
  if (p.log2_group < 2 || p.log2_group > 7) return cudaErrorInvalidValue;
  // bulk copies need 16-byte aligned sources (tile offsets are multiples of 16 B)
  auto a16 = [](const void* x) { return (reinterpret_cast<uintptr_t>(x) & 15u) == 0; };
  if (!a16(p.logits) || !a16(p.m_logits) || !a16(p.G) || !a16(p.W) || !a16(p.scales) ||
      !a16(p.m_scales) || (p.j0 && !a16(p.j0)) || ((p.n * 4) & 15))
    return cudaErrorInvalidValue;
  bool launched = false;
  cudaLaunchAttribute attr[1];
  pdl_attr(attr[0]);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid, 1, 1);
  cfg.blockDim = dim3(kEwThreads, 1, 1);
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  cudaError_t le = cudaSuccess;
  const cudaError_t e = with_relax(p.K, p.mode, [&](auto rx, auto sh) {
    using Rx = typename decltype(rx)::type;
    constexpr bool SH = decltype(sh)::value;
    with_plan<Rx::L>(plan, [&](auto pl) {
      using Plan = decltype(pl);
      const BwdStage S = stage_layout(Rx::L, Plan::kStageM, Plan::kStageGW, p.w_bf16, p.log2_group,
                                      p.scales_frozen, SH ? 1 : 0);
      cfg.dynamicSmemBytes = 2 * S.bytes;
      le = cudaLaunchKernelEx(&cfg, k_backward_staged<Rx, SH, Plan>, p, S);
      launched = true;
    });
  });
  if (e != cudaSuccess) return e;
  if (!launched) return cudaErrorInvalidValue;
  return le != cudaSuccess ? le : cudaGetLastError();
}

}  // namespace gsq
