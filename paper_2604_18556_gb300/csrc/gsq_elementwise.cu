// Elementwise kernels of the GSQ step (HBM-bound): initial state, forward
// (noise + tempered softmax + soft weight, Alg. 1), fused backward + Lion
// (+ the next step's forward), hard projection and packing.
//
// Data layout in HBM (n = E*R*C, flat index i = (e*R + r)*C + c):
//   logits, logit momenta : K planes of n fp32 ([K][E][R][C]), so every level is
//                           a unit-stride stream read with 128-bit loads;
//   scales, scale momenta : [n / G] fp32;  W, D : [n] (bf16 or fp32);  G : [n] fp32.
// Work split: one thread owns a quad of 4 consecutive weights (one float4 per
// plane); a scale group of G consecutive weights is G/4 adjacent lanes of one
// warp, so per-group sums are warp shuffles.  Grid-stride loops are warp-uniform.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <cstdlib>
#include <type_traits>

#include "gsq_internal.h"
#include "gsq_relax.cuh"
#include "gsq_tc.cuh"

namespace gsq {
namespace {

__device__ __forceinline__ void load_grid(const EwParams& P, float (&q)[kMaxLevels]) {
#pragma unroll
  for (int k = 0; k < kMaxLevels; ++k) q[k] = P.grid[k];
}

// Block-wide shared copy of the grid (local shift reads it with per-lane indices).
__device__ __forceinline__ void fill_shared_grid(const EwParams& P, float* sgrid) {
  if (threadIdx.x < kMaxLevels) sgrid[threadIdx.x] = P.grid[threadIdx.x];
  __syncthreads();
}


// Deterministic loss reduction: per-block double partials, summed in block
// order by the last block to finish (no device-side wait).
__device__ __forceinline__ void reduce_loss(float acc, const EwParams& P) {
  __shared__ double red[kEwThreads / 32];
  __shared__ bool is_last;
  double v = static_cast<double>(acc);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_down_sync(0xffffffffu, v, off);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
  __syncthreads();
  if (threadIdx.x == 0) {
    double s = 0.0;
    for (int w = 0; w < static_cast<int>(blockDim.x >> 5); ++w) s += red[w];
    P.loss_partials[blockIdx.x] = s;
    __threadfence();
    const unsigned int prev = atomicAdd(&P.flags->blocks_done, 1u);
    is_last = (prev == gridDim.x - 1);
  }
  __syncthreads();
  if (is_last) {  // the whole last block sums the partials, in a fixed order
    __threadfence();
    double s = 0.0;
    for (unsigned int b = threadIdx.x; b < gridDim.x; b += blockDim.x) s += __ldcg(P.loss_partials + b);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_down_sync(0xffffffffu, s, off);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
    __syncthreads();
    if (threadIdx.x == 0) {
      double t = 0.0;
      for (int w = 0; w < static_cast<int>(blockDim.x >> 5); ++w) t += red[w];
      if (P.loss_out) *P.loss_out = static_cast<float>(t);
      P.flags->blocks_done = 0u;
    }
  }
}

// ---------------------------------------------------------------------------
// Forward: D = s * w~ - W for step (t, tau, kappa); optional W^ export.
// Bytes per weight: read 4K (logits) + b_W, write 2 or 4 (D).
// ---------------------------------------------------------------------------
template <class Rx, bool kShift>
__global__ void __launch_bounds__(kEwThreads) k_forward(const EwParams P) {
  constexpr int K = Rx::L;
  float q[kMaxLevels];
  load_grid(P, q);
  __shared__ float sgrid[kMaxLevels];
  if (kShift) fill_shared_grid(P, sgrid);
  const PhiloxKeys& keys = P.keys;
  const int lane = threadIdx.x & 31;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t base = static_cast<int64_t>(blockIdx.x) * blockDim.x + (threadIdx.x & ~31);
       base < P.nq; base += stride) {
    const int64_t qi = base + lane;
    if (qi >= P.nq) continue;
    float l[K][4];
#pragma unroll
    for (int k = 0; k < K; ++k) {
      const float4 v = __ldcs(reinterpret_cast<const float4*>(P.logits + k * P.n) + qi);
      l[k][0] = v.x; l[k][1] = v.y; l[k][2] = v.z; l[k][3] = v.w;
    }
    float w[4];
    load_w4(P.W, qi, P.w_bf16, w);
    const float s = __ldg(P.scales + ((qi * 4) >> P.log2_group));
    const uint32_t j4 = kShift ? load_j0(P, qi) : 0u;
    float d[4], what[4];
#pragma unroll
    for (int pr = 0; pr < 2; ++pr) {
      float2 l2[K], h[K];
#pragma unroll
      for (int k = 0; k < K; ++k) l2[k] = make_float2(l[k][2 * pr], l[k][2 * pr + 1]);
      const Rx rx(q, sgrid, P.nlev, (j4 >> (16 * pr)) & 0xFFu, (j4 >> (16 * pr + 8)) & 0xFFu);
      Rx::noise(keys, P.t, static_cast<uint64_t>(qi) * 4 + 2 * pr, P.noise, h);
      const float2 wt = rx.value(l2, h, P.kappa_log2, P.inv_tau);
      // D = s w~ - W as one rounding per weight (identical in every kernel that forms D)
      const float2 wh = mul2(f2(s), wt);
      const float2 dd = fma2(f2(s), wt, make_float2(-w[2 * pr], -w[2 * pr + 1]));
      what[2 * pr] = wh.x; what[2 * pr + 1] = wh.y;
      d[2 * pr] = dd.x; d[2 * pr + 1] = dd.y;
    }
    store_d4(P.D, qi, P.d_bf16, d);
    if (P.what) reinterpret_cast<float4*>(P.what)[qi] = make_float4(what[0], what[1], what[2], what[3]);
  }
}

// ---------------------------------------------------------------------------
// Fused backward for step t: recompute the noise and the relaxation, loss
// partial 1/2 D*G, logit gradients (App. B), per-group scale gradient by
// warp shuffles, Lion in place; then (look-ahead) the forward of step t+1 from
// the updated registers.  Bytes per weight with look-ahead (L logits per
// weight): read 8L + 4 + b_W (+1 for j0), write 8L + 2 (D bf16).
// ---------------------------------------------------------------------------
// Blocks per SM the register budget aims for (measured best on GB300): two;
// three for the two-logit relaxations, which fit in 85 registers.
template <int K>
struct BwdOcc {
  static constexpr int value = 2;
};
template <>
struct BwdOcc<2> {
  static constexpr int value = 3;
};

// The per-quad body, shared by the kernel that loads its streams directly
// (k_backward) and the one that stages them through shared memory
// (k_backward_staged), so both do the same arithmetic.  l, m, gv, w, s, ms, j4
// hold the quad's inputs (m unused in export mode; gv zero for inactive lanes);
// l and m are updated in place.  Every lane of the warp calls it (the scale-group
// sums are shuffles).
template <class Rx, bool kExport, bool kShift, bool kAcc>
__device__ __forceinline__ void bwd_quad(const EwParams& P, const float (&q)[kMaxLevels],
                                         const float* sgrid, int lane, int seg, int64_t qi,
                                         bool active, float (&l)[Rx::L][4], float (&m)[Rx::L][4],
                                         float4 gv, const float (&w)[4], float s, float ms,
                                         uint32_t j4, float2& loss2) {
  constexpr int K = Rx::L;
  const PhiloxKeys& keys = P.keys;
  const int64_t qc = active ? qi : 0;
  const int64_t gidx = (qc * 4) >> P.log2_group;
  const float2 Gq[2] = {make_float2(gv.x, gv.y), make_float2(gv.z, gv.w)};
  float2 ds2 = f2(0.0f);
#pragma unroll
  for (int pr = 0; pr < 2; ++pr) {
    float2 l2[K], h[K];
#pragma unroll
    for (int k = 0; k < K; ++k) l2[k] = make_float2(l[k][2 * pr], l[k][2 * pr + 1]);
    Rx rx(q, sgrid, P.nlev, (j4 >> (16 * pr)) & 0xFFu, (j4 >> (16 * pr + 8)) & 0xFFu);
    Rx::noise(keys, P.t, static_cast<uint64_t>(qc) * 4 + 2 * pr, P.noise, h);
    const float2 wt = rx.relax(l2, h, P.kappa_log2, P.inv_tau);
    const float2 dd = fma2(f2(s), wt, make_float2(-w[2 * pr], -w[2 * pr + 1]));
    const float2 dj = make_float2(round_d(dd.x, P.d_bf16), round_d(dd.y, P.d_bf16));
    loss2 = fma2(mul2(f2(0.5f), dj), Gq[pr], loss2);
    ds2 = fma2(Gq[pr], wt, ds2);
    const float2 A = mul2(f2(P.kappa_over_tau * s), Gq[pr]);
#pragma unroll
    for (int k = 0; k < K; ++k) {
      // dL/dl_k = (kappa/tau) G s dw~/dl_k
      float2 dl = mul2(A, rx.dsoft(k));
      if (kAcc) {  // gradient accumulation: (this micro-batch + earlier ones) * scale
        const float2 a = reinterpret_cast<const float2*>(P.acc_in_l + k * P.n)[2 * qc + pr];
        dl = mul2(add2(dl, a), f2(P.acc_scale));
      }
      if (kExport) {
        m[k][2 * pr] = dl.x;
        m[k][2 * pr + 1] = dl.y;
      } else {
        // Lion, decoupled decay: c = b1 m + (1-b1) g; l <- l - lr wd l - lr sign(c);
        // m <- b2 m + (1-b2) g.  The decay is one fma on l (no rounded 1 - lr wd).
        const float2 mo = make_float2(m[k][2 * pr], m[k][2 * pr + 1]);
        const float2 c = fma2(f2(P.b1), mo, mul2(f2(1.0f - P.b1), dl));
        const float2 ln = add2(fma2(f2(-P.lrwd_l), l2[k], l2[k]),
                               make_float2(-lr_sign(P.lr_l, c.x), -lr_sign(P.lr_l, c.y)));
        const float2 mn = fma2(f2(P.b2), mo, mul2(f2(1.0f - P.b2), dl));
        l[k][2 * pr] = ln.x; l[k][2 * pr + 1] = ln.y;
        m[k][2 * pr] = mn.x; m[k][2 * pr + 1] = mn.y;
      }
    }
  }
  float ds = group_sum(ds2.x + ds2.y, seg);  // dL/ds_g = sum_{c in g} G_c w~_c
  if (kAcc && P.acc_in_s) ds = (ds + P.acc_in_s[gidx]) * P.acc_scale;

  if (kExport) {
    if (kAcc) __syncwarp();  // every lane has read acc_in_s before its group leader rewrites it
    if (active) {
      if (P.grad_logits) {
#pragma unroll
        for (int k = 0; k < K; ++k)
          reinterpret_cast<float4*>(P.grad_logits + k * P.n)[qi] =
              make_float4(m[k][0], m[k][1], m[k][2], m[k][3]);
      }
      if (P.grad_scales && !P.scales_frozen && (lane & (seg - 1)) == 0) P.grad_scales[gidx] = ds;
    }
  } else {
    if (!P.scales_frozen) {
      const float c = fmaf(P.b1, ms, (1.0f - P.b1) * ds);
      s = fmaf(-P.lrwd_s, s, s) - lr_sign(P.lr_s, c);
      ms = fmaf(P.b2, ms, (1.0f - P.b2) * ds);
    }
    if (active) {
#pragma unroll
      for (int k = 0; k < K; ++k) {
        __stcs(reinterpret_cast<float4*>(P.logits + k * P.n) + qi,
               make_float4(l[k][0], l[k][1], l[k][2], l[k][3]));
        __stcs(reinterpret_cast<float4*>(P.m_logits + k * P.n) + qi,
               make_float4(m[k][0], m[k][1], m[k][2], m[k][3]));
      }
      if (!P.scales_frozen && (lane & (seg - 1)) == 0) {
        P.scales[gidx] = s;
        P.m_scales[gidx] = ms;
      }
    }
  }
  if (active) {
    if (P.lookahead) {
      // forward of the next pass from the (updated, or in export mode unchanged)
      // logits and scale (Alg. 1)
      float d[4];
#pragma unroll
      for (int pr = 0; pr < 2; ++pr) {
        float2 l2[K], h[K];
#pragma unroll
        for (int k = 0; k < K; ++k) l2[k] = make_float2(l[k][2 * pr], l[k][2 * pr + 1]);
        const Rx rx(q, sgrid, P.nlev, (j4 >> (16 * pr)) & 0xFFu, (j4 >> (16 * pr + 8)) & 0xFFu);
        Rx::noise(keys, P.t_next, static_cast<uint64_t>(qi) * 4 + 2 * pr, P.noise, h);
        const float2 wt = rx.value(l2, h, P.kappa_log2_next, P.inv_tau_next);
        const float2 dd = fma2(f2(s), wt, make_float2(-w[2 * pr], -w[2 * pr + 1]));
        d[2 * pr] = dd.x;
        d[2 * pr + 1] = dd.y;
      }
      store_d4(P.D, qi, P.d_bf16, d);
    }
  }
}

// Direct loads of quad qi's inputs.  Lanes past the end (only in the last warp)
// read quad 0 and take G = 0, so every value stays finite and their loss and
// scale-gradient terms vanish; nothing is stored for them.  A scale group is
// never split across active and inactive lanes.
template <int K, bool kExport, bool kShift>
__device__ __forceinline__ void bwd_load_global(const EwParams& P, int64_t qi, bool active,
                                                float (&l)[K][4], float (&m)[K][4], float4& gv,
                                                float (&w)[4], float& s, float& ms, uint32_t& j4) {
  const int64_t qc = active ? qi : 0;
  const int64_t gidx = (qc * 4) >> P.log2_group;
#pragma unroll
  for (int k = 0; k < K; ++k) {
    const float4 v = __ldcs(reinterpret_cast<const float4*>(P.logits + k * P.n) + qc);
    l[k][0] = v.x; l[k][1] = v.y; l[k][2] = v.z; l[k][3] = v.w;
  }
  if (!kExport) {
#pragma unroll
    for (int k = 0; k < K; ++k) {
      const float4 v = __ldcs(reinterpret_cast<const float4*>(P.m_logits + k * P.n) + qc);
      m[k][0] = v.x; m[k][1] = v.y; m[k][2] = v.z; m[k][3] = v.w;
    }
  }
  gv = __ldcs(reinterpret_cast<const float4*>(P.G) + qc);
  if (!active) gv = make_float4(0.f, 0.f, 0.f, 0.f);
  load_w4(P.W, qc, P.w_bf16, w);
  s = __ldg(P.scales + gidx);
  ms = 0.0f;
  if (!kExport && !P.scales_frozen) ms = __ldg(P.m_scales + gidx);
  j4 = kShift ? load_j0(P, qc) : 0u;
}

template <class Rx, bool kExport, bool kShift, bool kAcc>
__global__ void __launch_bounds__(kEwThreads, BwdOcc<Rx::L>::value) k_backward(const EwParams P) {
  constexpr int K = Rx::L;
  float q[kMaxLevels];
  load_grid(P, q);
  __shared__ float sgrid[kMaxLevels];
  if (kShift) fill_shared_grid(P, sgrid);
  const int lane = threadIdx.x & 31;
  const int seg = P.group >> 2;  // lanes per scale group
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  float2 loss2 = f2(0.0f);

  for (int64_t base = static_cast<int64_t>(blockIdx.x) * blockDim.x + (threadIdx.x & ~31);
       base < P.nq; base += stride) {
    const int64_t qi = base + lane;
    const bool active = qi < P.nq;
    float l[K][4], m[K][4], w[4];
    float4 gv;
    float s, ms;
    uint32_t j4;
    bwd_load_global<K, kExport, kShift>(P, qi, active, l, m, gv, w, s, ms, j4);
    bwd_quad<Rx, kExport, kShift, kAcc>(P, q, sgrid, lane, seg, qi, active, l, m, gv, w, s, ms,
                                        j4, loss2);
  }
  reduce_loss(loss2.x + loss2.y, P);
}

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
// Logit momenta are staged for L <= 5 logits, where two stages of two resident
// blocks fit in shared memory; otherwise they are loaded directly at the top of
// the iteration and arrive while the noise is drawn.  Stores stay direct.
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

// ---------------------------------------------------------------------------
// Initial state.  Group mode: s = absmax_g / max|q| (1 for an all-zero group);
// RTN code k0 = argmin_k |W/s - q_k| (lowest k on ties); logits = bias on k0.
// All decisions in fp32 with IEEE division, as the oracle takes them.
// ---------------------------------------------------------------------------
__device__ __forceinline__ int rtn_code(float w, float s, const float (&q)[kMaxLevels], int K,
                                        int zero_code) {
  if (s == 0.0f) return zero_code;
  const float x = __fdiv_rn(w, s);
  int best = 0;
  float bd = fabsf(x - q[0]);
  for (int k = 1; k < K; ++k) {
    const float dk = fabsf(x - q[k]);
    if (dk < bd) {
      bd = dk;
      best = k;
    }
  }
  return best;
}

struct InitConsts {
  float q[kMaxLevels];
  float qmax;
  int zero_code;
};

__device__ __forceinline__ InitConsts init_consts(const InitParams& P) {
  InitConsts c;
  c.qmax = 0.0f;
  c.zero_code = 0;
  float zmin = INFINITY;
  for (int k = 0; k < kMaxLevels; ++k) c.q[k] = P.grid[k];
  for (int k = 0; k < P.K; ++k) {
    c.qmax = fmaxf(c.qmax, fabsf(c.q[k]));
    if (fabsf(c.q[k]) < zmin) {
      zmin = fabsf(c.q[k]);
      c.zero_code = k;
    }
  }
  return c;
}

// Logits of a quad: init_bias on the RTN level (or, with local shift, on the
// delta = 0 logit, with the RTN index stored as j0); momenta 0.
__device__ __forceinline__ void write_init_quad(const InitParams& P, int64_t qi, const int (&code)[4]) {
  const uint32_t c4 = static_cast<uint32_t>(code[0]) | (static_cast<uint32_t>(code[1]) << 8) |
                      (static_cast<uint32_t>(code[2]) << 16) | (static_cast<uint32_t>(code[3]) << 24);
  if (P.j0) reinterpret_cast<uint32_t*>(P.j0)[qi] = c4;
  if (P.code0) reinterpret_cast<uint32_t*>(P.code0)[qi] = c4;
  if (P.mask_sign) {
    // Eq. 3 on the RTN code (0, 1, 2 for -a, 0, a), times init_bias:
    // l_m = +b if the code is nonzero else -b; l_b = +b, -b or 0 by its sign
    const float b = P.init_bias;
    float lm[4], lb[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      lm[j] = code[j] != 1 ? b : -b;
      lb[j] = code[j] == 2 ? b : (code[j] == 0 ? -b : 0.0f);
    }
    reinterpret_cast<float4*>(P.logits)[qi] = make_float4(lm[0], lm[1], lm[2], lm[3]);
    reinterpret_cast<float4*>(P.logits + P.n)[qi] = make_float4(lb[0], lb[1], lb[2], lb[3]);
    for (int k = 0; k < 2; ++k)
      reinterpret_cast<float4*>(P.m_logits + k * P.n)[qi] = make_float4(0.f, 0.f, 0.f, 0.f);
    return;
  }
  const int logits = P.j0 ? 5 : P.K;
  for (int k = 0; k < logits; ++k) {
    float4 v;
    if (P.j0) {
      const float b = k == 2 ? P.init_bias : 0.0f;
      v = make_float4(b, b, b, b);
    } else {
      v.x = code[0] == k ? P.init_bias : 0.0f;
      v.y = code[1] == k ? P.init_bias : 0.0f;
      v.z = code[2] == k ? P.init_bias : 0.0f;
      v.w = code[3] == k ? P.init_bias : 0.0f;
    }
    reinterpret_cast<float4*>(P.logits + k * P.n)[qi] = v;
    reinterpret_cast<float4*>(P.m_logits + k * P.n)[qi] = make_float4(0.f, 0.f, 0.f, 0.f);
  }
}

__global__ void __launch_bounds__(kEwThreads) k_init_group(const InitParams P) {
  const InitConsts c = init_consts(P);
  const int lane = threadIdx.x & 31;
  const int seg = P.group >> 2;
  const int64_t nq = P.n >> 2;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  int log2g = 0;
  while ((1 << log2g) < P.group) ++log2g;
  for (int64_t base = static_cast<int64_t>(blockIdx.x) * blockDim.x + (threadIdx.x & ~31);
       base < nq; base += stride) {
    const int64_t qi = base + lane;
    const bool active = qi < nq;
    float w[4] = {0.f, 0.f, 0.f, 0.f};
    if (active) load_w4(P.W, qi, P.w_bf16, w);
    float amax = fmaxf(fmaxf(fabsf(w[0]), fabsf(w[1])), fmaxf(fabsf(w[2]), fabsf(w[3])));
    for (int off = 1; off < seg; off <<= 1)
      amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, off));
    if (!active) continue;
    const float s = amax == 0.0f ? 1.0f : __fdiv_rn(amax, c.qmax);
    int code[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) code[j] = rtn_code(w[j], s, c.q, P.K, c.zero_code);
    write_init_quad(P, qi, code);
    if ((lane & (seg - 1)) == 0) {
      const int64_t gi = (qi * 4) >> log2g;
      P.scales[gi] = s;
      P.m_scales[gi] = 0.0f;
    }
  }
}

// K-Quant-like two-level scales: one warp per 256-weight super-block, lane l
// owns weights 8l..8l+7 (sub-block l/2).  s_j = absmax_16 / max|q|;
// d = fp16_rne(max_j s_j / 31); sc_j = clamp(rne(s_j / d), -32, 31) (0 if d = 0);
// effective scale d*sc_j (exact in fp32).
__global__ void __launch_bounds__(kEwThreads) k_init_kquant(const InitParams P) {
  const InitConsts c = init_consts(P);
  const int lane = threadIdx.x & 31;
  const int64_t nsb = P.n / kSuperBlock;
  const int64_t warps = static_cast<int64_t>(gridDim.x) * (blockDim.x >> 5);
  for (int64_t sb = static_cast<int64_t>(blockIdx.x) * (blockDim.x >> 5) + (threadIdx.x >> 5);
       sb < nsb; sb += warps) {
    const int64_t q0 = sb * (kSuperBlock / 4) + 2 * lane;  // first of this lane's two quads
    float w[8];
    {
      float a[4], b[4];
      load_w4(P.W, q0, P.w_bf16, a);
      load_w4(P.W, q0 + 1, P.w_bf16, b);
      for (int j = 0; j < 4; ++j) {
        w[j] = a[j];
        w[4 + j] = b[j];
      }
    }
    float amax = 0.0f;
    for (int j = 0; j < 8; ++j) amax = fmaxf(amax, fabsf(w[j]));
    amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, 1));
    const float sj = __fdiv_rn(amax, c.qmax);
    float smax = sj;
    for (int off = 2; off < 32; off <<= 1) smax = fmaxf(smax, __shfl_xor_sync(0xffffffffu, smax, off));
    const __half dh = __float2half_rn(__fdiv_rn(smax, 31.0f));
    const float d = __half2float(dh);
    int sc = 0;
    if (d > 0.0f) sc = static_cast<int>(fminf(fmaxf(rintf(__fdiv_rn(sj, d)), -32.0f), 31.0f));
    const float s = d * static_cast<float>(sc);
    int code[2][4];
    for (int j = 0; j < 8; ++j) code[j >> 2][j & 3] = rtn_code(w[j], s, c.q, P.K, c.zero_code);
    write_init_quad(P, q0, code[0]);
    write_init_quad(P, q0 + 1, code[1]);
    if ((lane & 1) == 0) {
      const int64_t sub = sb * (kSuperBlock / kSubBlock) + (lane >> 1);
      P.scales[sub] = s;
      P.m_scales[sub] = 0.0f;
      P.kq_sc[sub] = static_cast<int8_t>(sc);
    }
    if (lane == 0) P.kq_d[sb] = __half_as_ushort(dh);
  }
}

// Warm start from supplied codes (Eq. 3-4, App. A): l = sigma (eps + alpha l_prior)
// per logit plane, momenta 0; one quad of weights per thread and iteration.
__device__ __forceinline__ float prior_logit(const InitCodesParams& P, int k, int c) {
  if (P.mode == GSQ_PARAM_MASK_SIGN) {          // Eq. 3
    if (k == 0) return c != 1 ? 1.0f : -1.0f;
    return c == 2 ? 1.0f : (c == 0 ? -1.0f : 0.0f);
  }
  if (P.mode == GSQ_PARAM_SHIFT5) {             // -(d^2)/2 for d = k - 2, mean -1 removed
    const float d = static_cast<float>(k - 2);
    return 1.0f - 0.5f * d * d;
  }
  // -(q_k - q_c)^2 / 2 minus its mean over the K levels
  const float mu = P.grid[c];
  float mean = 0.0f;
  for (int j = 0; j < P.K; ++j) {
    const float e = P.grid[j] - mu;
    mean += e * e;
  }
  mean = -0.5f * mean / static_cast<float>(P.K);
  const float e = P.grid[k] - mu;
  return -0.5f * e * e - mean;
}

__global__ void __launch_bounds__(kEwThreads) k_init_from_codes(const InitCodesParams P) {
  const int L = P.mode == GSQ_PARAM_SHIFT5 ? 5 : (P.mode == GSQ_PARAM_MASK_SIGN ? 2 : P.K);
  const int64_t nq = P.n >> 2;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t qi = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; qi < nq; qi += stride) {
    uint32_t c4 = reinterpret_cast<const uint32_t*>(P.codes)[qi];
    int c[4];
    uint32_t clamped = 0;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      c[j] = min(static_cast<int>((c4 >> (8 * j)) & 0xFFu), P.K - 1);
      clamped |= static_cast<uint32_t>(c[j]) << (8 * j);
    }
    if (P.j0) reinterpret_cast<uint32_t*>(P.j0)[qi] = clamped;
    if (P.code0) reinterpret_cast<uint32_t*>(P.code0)[qi] = clamped;
    for (int k = 0; k < L; ++k) {
      float4 e = make_float4(0.f, 0.f, 0.f, 0.f);
      if (P.eps) e = __ldcs(reinterpret_cast<const float4*>(P.eps + k * P.n) + qi);
      float4 v;
      v.x = P.sigma * fmaf(P.alpha, prior_logit(P, k, c[0]), e.x);
      v.y = P.sigma * fmaf(P.alpha, prior_logit(P, k, c[1]), e.y);
      v.z = P.sigma * fmaf(P.alpha, prior_logit(P, k, c[2]), e.z);
      v.w = P.sigma * fmaf(P.alpha, prior_logit(P, k, c[3]), e.w);
      reinterpret_cast<float4*>(P.logits + k * P.n)[qi] = v;
      reinterpret_cast<float4*>(P.m_logits + k * P.n)[qi] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
  }
}

__global__ void k_nonfinite(const void* x, int64_t count, int bf16, unsigned int* counter) {
  unsigned int bad = 0;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < count; i += stride) {
    float v;
    if (bf16)
      v = __bfloat162float(reinterpret_cast<const __nv_bfloat16*>(x)[i]);
    else
      v = reinterpret_cast<const float*>(x)[i];
    bad += isfinite(v) ? 0u : 1u;
  }
  for (int off = 16; off > 0; off >>= 1) bad += __shfl_down_sync(0xffffffffu, bad, off);
  if ((threadIdx.x & 31) == 0 && bad) atomicAdd(counter, bad);
}

// ---------------------------------------------------------------------------
// Hard projection: k* = argmax_k l_k (lowest k on ties), margin l_(1) - l_(2).
// ---------------------------------------------------------------------------
__device__ __forceinline__ void argmax_margin(const float* logits, int64_t n, int K, int64_t i,
                                              int& code, float& margin) {
  float best = __ldcs(logits + i), second = -INFINITY;
  code = 0;
  for (int k = 1; k < K; ++k) {
    const float v = __ldcs(logits + k * n + i);
    if (v > best) {
      second = best;
      best = v;
      code = k;
    } else if (v > second) {
      second = v;
    }
  }
  margin = best - second;
}

// Grid code of logit index k: k itself, or clip(j0 + k - 2) with local shift.
__device__ __forceinline__ int grid_code(int k, const uint8_t* j0, int64_t i, int nlev) {
  return j0 ? min(max(static_cast<int>(j0[i]) + k - 2, 0), nlev - 1) : k;
}

// Mask x sign hard rule (Alg. 2): m = [l_m >= 0], b = 2 [l_b >= 0] - 1; code
// 1 (zero) when the mask is off, else 2 or 0 by the sign.  Margin: the top-two
// logit gap 2|l| of every instance that decides the code.
__device__ __forceinline__ void mask_sign_code(float lm, float lb, int& code, float& margin) {
  const bool m = lm >= 0.0f;
  code = m ? (lb >= 0.0f ? 2 : 0) : 1;
  margin = m ? fminf(2.0f * fabsf(lm), 2.0f * fabsf(lb)) : 2.0f * fabsf(lm);
}

// Final code and margin of weight i under any parameterisation.
template <class P_>
__device__ __forceinline__ void decide(const P_& P, int64_t i, int& code, float& margin) {
  if (P.mask_sign) {
    mask_sign_code(__ldcs(P.logits + i), __ldcs(P.logits + P.n + i), code, margin);
    return;
  }
  argmax_margin(P.logits, P.n, P.K, i, code, margin);
  code = grid_code(code, P.j0, i, P.nlev);
}

__global__ void __launch_bounds__(kEwThreads) k_project(const ProjectParams P) {
  const int64_t nq = P.n >> 2;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t qi = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; qi < nq; qi += stride) {
    if (P.mask_sign) {
      const float4 a = __ldcs(reinterpret_cast<const float4*>(P.logits) + qi);
      const float4 b = __ldcs(reinterpret_cast<const float4*>(P.logits + P.n) + qi);
      int c[4];
      float mg[4];
      mask_sign_code(a.x, b.x, c[0], mg[0]);
      mask_sign_code(a.y, b.y, c[1], mg[1]);
      mask_sign_code(a.z, b.z, c[2], mg[2]);
      mask_sign_code(a.w, b.w, c[3], mg[3]);
      if (P.codes)
        reinterpret_cast<uint32_t*>(P.codes)[qi] =
            static_cast<uint32_t>(c[0]) | (static_cast<uint32_t>(c[1]) << 8) |
            (static_cast<uint32_t>(c[2]) << 16) | (static_cast<uint32_t>(c[3]) << 24);
      if (P.margin) reinterpret_cast<float4*>(P.margin)[qi] = make_float4(mg[0], mg[1], mg[2], mg[3]);
      continue;
    }
    float best[4], second[4];
    int code[4] = {0, 0, 0, 0};
    {
      const float4 v = __ldcs(reinterpret_cast<const float4*>(P.logits) + qi);
      best[0] = v.x; best[1] = v.y; best[2] = v.z; best[3] = v.w;
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) second[j] = -INFINITY;
    for (int k = 1; k < P.K; ++k) {
      const float4 v4 = __ldcs(reinterpret_cast<const float4*>(P.logits + k * P.n) + qi);
      const float v[4] = {v4.x, v4.y, v4.z, v4.w};
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        if (v[j] > best[j]) {
          second[j] = best[j];
          best[j] = v[j];
          code[j] = k;
        } else if (v[j] > second[j]) {
          second[j] = v[j];
        }
      }
    }
    if (P.j0) {
      const uint32_t j4 = reinterpret_cast<const uint32_t*>(P.j0)[qi];
#pragma unroll
      for (int j = 0; j < 4; ++j)
        code[j] = min(max(static_cast<int>((j4 >> (8 * j)) & 0xFFu) + code[j] - 2, 0), P.nlev - 1);
    }
    if (P.codes) {
      const uint32_t packed = static_cast<uint32_t>(code[0]) | (static_cast<uint32_t>(code[1]) << 8) |
                              (static_cast<uint32_t>(code[2]) << 16) | (static_cast<uint32_t>(code[3]) << 24);
      reinterpret_cast<uint32_t*>(P.codes)[qi] = packed;
    }
    if (P.margin)
      reinterpret_cast<float4*>(P.margin)[qi] =
          make_float4(best[0] - second[0], best[1] - second[1], best[2] - second[2], best[3] - second[3]);
  }
}

// ---------------------------------------------------------------------------
// Packing.  One warp per chunk of 32 consecutive weights: lane j projects weight
// j of the chunk and contributes its code at bit b*j of the chunk's b-word
// little-endian stream; the words are OR-reduced across the warp.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t stream_word(uint32_t code, int bits, int lane, int word) {
  const int shift = bits * lane - 32 * word;  // position of this code inside `word`
  if (shift >= 32 || shift <= -bits) return 0u;
  return shift >= 0 ? (code << shift) : (code >> (-shift));
}

__global__ void __launch_bounds__(kEwThreads) k_pack_group(const PackParams P) {
  const int lane = threadIdx.x & 31;
  const int bits = P.nlev <= 4 ? 2 : 3;
  const int64_t nchunks = (P.n + 31) / 32;
  const int64_t warps = static_cast<int64_t>(gridDim.x) * (blockDim.x >> 5);
  uint32_t* words = reinterpret_cast<uint32_t*>(P.out);
  for (int64_t ch = static_cast<int64_t>(blockIdx.x) * (blockDim.x >> 5) + (threadIdx.x >> 5);
       ch < nchunks; ch += warps) {
    const int64_t i = ch * 32 + lane;
    uint32_t code = 0;
    if (i < P.n) {
      int c;
      float mg;
      decide(P, i, c, mg);
      code = static_cast<uint32_t>(c);
    }
    for (int wd = 0; wd < bits; ++wd) {
      const uint32_t v = __reduce_or_sync(0xffffffffu, stream_word(code, bits, lane, wd));
      if (lane == wd) words[ch * bits + wd] = v;
    }
  }
  // fp16 (round-to-nearest-even) group scales after the padded code section
  uint16_t* sc = reinterpret_cast<uint16_t*>(P.out + P.code_bytes);
  const int64_t ng = P.n / P.group;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t g = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; g < ng; g += stride)
    sc[g] = __half_as_ushort(__float2half_rn(P.scales[g]));
  // zero the padding words of the code section
  const int64_t used = nchunks * bits;
  for (int64_t wi = used + static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
       wi < P.code_bytes / 4; wi += stride)
    words[wi] = 0u;
}

__global__ void __launch_bounds__(kEwThreads) k_pack_kquant(const PackParams P) {
  __shared__ uint32_t rec[kEwThreads / 32][28];
  const int lane = threadIdx.x & 31;
  const int wib = threadIdx.x >> 5;
  const int64_t nsb = P.n / kSuperBlock;
  const int64_t warps = static_cast<int64_t>(gridDim.x) * (blockDim.x >> 5);
  for (int64_t sb = static_cast<int64_t>(blockIdx.x) * (blockDim.x >> 5) + wib; sb < nsb; sb += warps) {
    for (int ch = 0; ch < 8; ++ch) {
      int c;
      float mg;
      const int64_t wi = sb * kSuperBlock + ch * 32 + lane;
      decide(P, wi, c, mg);
      for (int wd = 0; wd < 3; ++wd) {
        const uint32_t v = __reduce_or_sync(0xffffffffu, stream_word(static_cast<uint32_t>(c), 3, lane, wd));
        if (lane == wd) rec[wib][ch * 3 + wd] = v;
      }
    }
    uint32_t s6 = 0;
    if (lane < 16) s6 = static_cast<uint32_t>(static_cast<int>(P.kq_sc[sb * 16 + lane]) + 32) & 63u;
    for (int wd = 0; wd < 3; ++wd) {
      const uint32_t v = __reduce_or_sync(0xffffffffu, lane < 16 ? stream_word(s6, 6, lane, wd) : 0u);
      if (lane == wd) rec[wib][24 + wd] = v;
    }
    if (lane == 0) rec[wib][27] = static_cast<uint32_t>(P.kq_d[sb]);
    __syncwarp();
    const uint8_t* bytes = reinterpret_cast<const uint8_t*>(rec[wib]);
    uint8_t* dst = P.out + sb * kKqRecord;
    for (int b = lane; b < kKqRecord; b += 32) dst[b] = bytes[b];
    __syncwarp();
  }
}

// ---------------------------------------------------------------------------
// Diagnostics of the current logits (no noise): histogram of |code - initial
// code|, histogram of top-two margins (bins split at 1e-6 ... 10, compared in
// fp32), and per-block sums of the max probability of softmax(kappa l / tau)
// (of the three-value distribution for mask x sign).  Counts are integers, so
// their atomics commute; the probability sums go out per block.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kEwThreads) k_diagnose(const DiagParams P) {
  __shared__ unsigned int hist[kDiagShiftBins + kDiagMarginBins];
  __shared__ double red[kEwThreads / 32];
  for (int i = threadIdx.x; i < kDiagShiftBins + kDiagMarginBins; i += blockDim.x) hist[i] = 0u;
  __syncthreads();
  const float edges[kDiagMarginBins - 1] = {1e-6f, 1e-5f, 1e-4f, 1e-3f, 1e-2f, 1e-1f, 1.0f, 10.0f};
  double acc = 0.0;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < P.n; i += stride) {
    int code;
    float mg;
    decide(P, i, code, mg);
    const int d = abs(code - static_cast<int>(P.code0[i]));
    atomicAdd(&hist[d < kDiagShiftBins ? d : kDiagShiftBins - 1], 1u);
    int b = 0;
#pragma unroll
    for (int e = 0; e < kDiagMarginBins - 1; ++e) b += mg >= edges[e] ? 1 : 0;
    atomicAdd(&hist[kDiagShiftBins + b], 1u);
    // fp32 arithmetic (a monitoring statistic), double accumulation
    const float kot = static_cast<float>(P.kappa_over_tau);
    float pmax;
    if (P.mask_sign) {
      const float pm = 1.0f / (1.0f + expf(-2.0f * kot * P.logits[i]));
      const float pb = 1.0f / (1.0f + expf(-2.0f * kot * P.logits[P.n + i]));
      pmax = fmaxf(fmaxf(pm * (1.0f - pb), 1.0f - pm), pm * pb);
    } else {
      float lmax = P.logits[i];
      for (int k = 1; k < P.K; ++k) lmax = fmaxf(lmax, P.logits[k * P.n + i]);
      float sum = 0.0f;
      for (int k = 0; k < P.K; ++k) sum += expf(kot * (P.logits[k * P.n + i] - lmax));
      pmax = 1.0f / sum;
    }
    acc += static_cast<double>(pmax);
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) acc += __shfl_down_sync(0xffffffffu, acc, off);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    double s = 0.0;
    for (int w = 0; w < static_cast<int>(blockDim.x >> 5); ++w) s += red[w];
    P.partials[blockIdx.x] = s;
  }
  for (int i = threadIdx.x; i < kDiagShiftBins + kDiagMarginBins; i += blockDim.x)
    if (hist[i]) atomicAdd(P.hist + i, static_cast<unsigned long long>(hist[i]));
}

template <class Rx, bool kShift>
void set_max_smem_carveout() {
  const auto attr = cudaFuncAttributePreferredSharedMemoryCarveout;
  cudaFuncSetAttribute(k_forward<Rx, kShift>, attr, 0);
  cudaFuncSetAttribute(k_backward<Rx, false, kShift, false>, attr, 0);
  cudaFuncSetAttribute(k_backward<Rx, true, kShift, false>, attr, 0);
  cudaFuncSetAttribute(k_backward<Rx, false, kShift, true>, attr, 0);
  cudaFuncSetAttribute(k_backward<Rx, true, kShift, true>, attr, 0);
}

int grid_for(const void* fn, int num_sms, int threads) {
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, threads, 0) != cudaSuccess ||
      per_sm < 1)
    per_sm = 1;
  return per_sm * num_sms;
}

}  // namespace


int ew_grid_size(int K, int which, int num_sms, int mode) {
  int g = num_sms;
  with_relax(K, mode, [&](auto rx, auto sh) {
    using Rx = typename decltype(rx)::type;
    constexpr bool SH = decltype(sh)::value;
    set_max_smem_carveout<Rx, SH>();
    g = which == 0 ? grid_for(reinterpret_cast<const void*>(k_forward<Rx, SH>), num_sms, kEwThreads)
                   : grid_for(reinterpret_cast<const void*>(k_backward<Rx, false, SH, false>), num_sms,
                              kEwThreads);
  });
  return g;
}

cudaError_t launch_forward(const EwParams& p, int grid, cudaStream_t s) {
  const cudaError_t e = with_relax(p.K, p.mode, [&](auto rx, auto sh) {
    using Rx = typename decltype(rx)::type;
    k_forward<Rx, decltype(sh)::value><<<grid, kEwThreads, 0, s>>>(p);
  });
  return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_backward(const EwParams& p, int grid, cudaStream_t s) {
  const bool export_mode = (p.grad_logits != nullptr) || (p.grad_scales != nullptr);
  const bool acc = p.acc_in_l != nullptr;
  const cudaError_t e = with_relax(p.K, p.mode, [&](auto rx, auto sh) {
    using Rx = typename decltype(rx)::type;
    constexpr bool SH = decltype(sh)::value;
    if (export_mode)
      acc ? k_backward<Rx, true, SH, true><<<grid, kEwThreads, 0, s>>>(p)
          : k_backward<Rx, true, SH, false><<<grid, kEwThreads, 0, s>>>(p);
    else
      acc ? k_backward<Rx, false, SH, true><<<grid, kEwThreads, 0, s>>>(p)
          : k_backward<Rx, false, SH, false><<<grid, kEwThreads, 0, s>>>(p);
  });
  return e != cudaSuccess ? e : cudaGetLastError();
}

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

cudaError_t launch_backward_staged(const EwParams& p, int grid, int plan, cudaStream_t s) {
  if (p.grad_logits || p.grad_scales || p.acc_in_l || p.acc_in_s) return cudaErrorInvalidValue;
  if (p.log2_group < 2 || p.log2_group > 7) return cudaErrorInvalidValue;
  // bulk copies need 16-byte aligned sources (tile offsets are multiples of 16 B)
  auto a16 = [](const void* x) { return (reinterpret_cast<uintptr_t>(x) & 15u) == 0; };
  if (!a16(p.logits) || !a16(p.m_logits) || !a16(p.G) || !a16(p.W) || !a16(p.scales) ||
      !a16(p.m_scales) || (p.j0 && !a16(p.j0)) || ((p.n * 4) & 15))
    return cudaErrorInvalidValue;
  bool launched = false;
  const cudaError_t e = with_relax(p.K, p.mode, [&](auto rx, auto sh) {
    using Rx = typename decltype(rx)::type;
    constexpr bool SH = decltype(sh)::value;
    with_plan<Rx::L>(plan, [&](auto pl) {
      using Plan = decltype(pl);
      const BwdStage S = stage_layout(Rx::L, Plan::kStageM, Plan::kStageGW, p.w_bf16, p.log2_group,
                                      p.scales_frozen, SH ? 1 : 0);
      k_backward_staged<Rx, SH, Plan><<<grid, kEwThreads, 2 * S.bytes, s>>>(p, S);
      launched = true;
    });
  });
  if (e != cudaSuccess) return e;
  if (!launched) return cudaErrorInvalidValue;
  return cudaGetLastError();
}

cudaError_t launch_init_state(const InitParams& p, int num_sms, cudaStream_t s) {
  if (p.kquant) {
    const int64_t nsb = p.n / kSuperBlock;
    const int64_t blocks = (nsb + (kEwThreads / 32) - 1) / (kEwThreads / 32);
    const int grid = static_cast<int>(blocks < 16LL * num_sms ? blocks : 16LL * num_sms);
    k_init_kquant<<<grid > 0 ? grid : 1, kEwThreads, 0, s>>>(p);
  } else {
    const int64_t blocks = ((p.n >> 2) + kEwThreads - 1) / kEwThreads;
    const int grid = static_cast<int>(blocks < 16LL * num_sms ? blocks : 16LL * num_sms);
    k_init_group<<<grid > 0 ? grid : 1, kEwThreads, 0, s>>>(p);
  }
  return cudaGetLastError();
}

cudaError_t launch_init_from_codes(const InitCodesParams& p, int num_sms, cudaStream_t s) {
  const int64_t blocks = ((p.n >> 2) + kEwThreads - 1) / kEwThreads;
  const int grid = static_cast<int>(blocks < 8LL * num_sms ? blocks : 8LL * num_sms);
  k_init_from_codes<<<grid > 0 ? grid : 1, kEwThreads, 0, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_nonfinite_scan(const void* x, int64_t count, int is_bf16, unsigned int* counter,
                                  cudaStream_t s) {
  if (count <= 0) return cudaSuccess;
  const int64_t blocks = (count + 255) / 256;
  const int grid = static_cast<int>(blocks < 4096 ? blocks : 4096);
  k_nonfinite<<<grid, 256, 0, s>>>(x, count, is_bf16, counter);
  return cudaGetLastError();
}

cudaError_t launch_diagnose(const DiagParams& p, int grid, cudaStream_t s) {
  k_diagnose<<<grid, kEwThreads, 0, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_project(const ProjectParams& p, int num_sms, cudaStream_t s) {
  const int64_t blocks = ((p.n >> 2) + kEwThreads - 1) / kEwThreads;
  const int grid = static_cast<int>(blocks < 8LL * num_sms ? blocks : 8LL * num_sms);
  k_project<<<grid > 0 ? grid : 1, kEwThreads, 0, s>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_pack(const PackParams& p, int num_sms, cudaStream_t s) {
  const int grid = 8 * num_sms;
  if (p.kquant)
    k_pack_kquant<<<grid, kEwThreads, 0, s>>>(p);
  else
    k_pack_group<<<grid, kEwThreads, 0, s>>>(p);
  return cudaGetLastError();
}

}  // namespace gsq
