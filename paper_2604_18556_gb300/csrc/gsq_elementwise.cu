// Elementwise kernels of the GSQ step (HBM-bound): initial state, forward
// (noise + tempered softmax + soft weight, Alg. 1), hard projection, packing and
// diagnostics.  The fused backward + Lion (+ the next step's forward) is in
// gsq_backward.cu and gsq_staged.cu.
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

#include <type_traits>

#include "gsq_backward.cuh"
#include "gsq_internal.h"
#include "gsq_relax.cuh"

namespace gsq {
namespace {

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
      Rx::noise(keys, P.t, P.index_base + static_cast<uint64_t>(qi) * 4 + 2 * pr, P.noise, h);
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
void set_forward_carveout() {
  cudaFuncSetAttribute(k_forward<Rx, kShift>, cudaFuncAttributePreferredSharedMemoryCarveout, 0);
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
  if (which != 0) return ew_backward_grid(K, num_sms, mode);
  int g = num_sms;
  with_relax(K, mode, [&](auto rx, auto sh) {
    using Rx = typename decltype(rx)::type;
    constexpr bool SH = decltype(sh)::value;
    set_forward_carveout<Rx, SH>();
    g = grid_for(reinterpret_cast<const void*>(k_forward<Rx, SH>), num_sms, kEwThreads);
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
