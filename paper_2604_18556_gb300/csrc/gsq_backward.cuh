// Device code shared by the elementwise kernels (gsq_elementwise.cu) and the two
// fused backward kernels (gsq_backward.cu: direct loads; gsq_staged.cu: streams
// staged through shared memory): the grid constants, the deterministic loss
// reduction, and the per-quad body of the fused backward (noise, relaxation,
// App. B gradients, Lion, look-ahead forward).  Internal linkage: every
// translation unit that includes it gets its own copy.
//
// Data layout in HBM (n = E*R*C, flat index i = (e*R + r)*C + c):
//   logits, logit momenta : K planes of n fp32 ([K][E][R][C]), so every level is
//                           a unit-stride stream read with 128-bit loads;
//   scales, scale momenta : [n / G] fp32;  W, D : [n] (bf16 or fp32);  G : [n] fp32.
// Work split: one thread owns a quad of 4 consecutive weights (one float4 per
// plane); a scale group of G consecutive weights is G/4 adjacent lanes of one
// warp, so per-group sums are warp shuffles.  Grid-stride loops are warp-uniform.
#pragma once

#include <cuda_bf16.h>

#include "gsq_internal.h"
#include "gsq_relax.cuh"

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
    Rx::noise(keys, P.t, P.index_base + static_cast<uint64_t>(qc) * 4 + 2 * pr, P.noise, h);
    const float2 wt = rx.relax(l2, h, P.kappa_log2, P.inv_tau);
    const float2 dd = fma2(f2(s), wt, make_float2(-w[2 * pr], -w[2 * pr + 1]));
    const float2 dj = make_float2(round_d(dd.x, P.d_bf16), round_d(dd.y, P.d_bf16));
    loss2 = fma2(mul2(f2(0.5f), dj), Gq[pr], loss2);
    ds2 = fma2(Gq[pr], wt, ds2);
    float2 A = mul2(f2(P.kappa_over_tau * s), Gq[pr]);
    if (Rx::kScaled) A = mul2(A, rx.dscale());
    // Lion mixes (1 - b1) and (1 - b2) of each gradient into c and the momentum:
    // both factors ride on A, one product per pair instead of one per logit
    const float2 A1 = mul2(A, f2(1.0f - P.b1)), A2 = mul2(A, f2(1.0f - P.b2));
#pragma unroll
    for (int k = 0; k < K; ++k) {
      // dL/dl_k = (kappa/tau) G s dw~/dl_k
      const float2 dk = rx.dsoft(k);
      float2 dl = mul2(A, dk);
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
        const float2 c = kAcc ? fma2(f2(P.b1), mo, mul2(f2(1.0f - P.b1), dl))
                              : fma2(f2(P.b1), mo, mul2(A1, dk));
        const float2 ln = add2(fma2(f2(-P.lrwd_l), l2[k], l2[k]),
                               make_float2(-lr_sign(P.lr_l, c.x), -lr_sign(P.lr_l, c.y)));
        const float2 mn = kAcc ? fma2(f2(P.b2), mo, mul2(f2(1.0f - P.b2), dl))
                               : fma2(f2(P.b2), mo, mul2(A2, dk));
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
        Rx::noise(keys, P.t_next, P.index_base + static_cast<uint64_t>(qi) * 4 + 2 * pr, P.noise, h);
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

}  // namespace
}  // namespace gsq
