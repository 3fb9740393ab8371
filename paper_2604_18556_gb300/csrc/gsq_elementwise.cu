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

#include <type_traits>

#include "gsq_internal.h"

namespace gsq {
namespace {

// ---------------------------------------------------------------------------
// Counter-based Gumbel noise (Alg. 1 draw; resampled every step, §3.3).
// Philox4x32-10 from its definition (Salmon, Moraes, Dror, Shaw, SC'11):
// S-box multipliers 0xD2511F53 / 0xCD9E8D57, Weyl key increments 0x9E3779B9 /
// 0xBB67AE85.  Counter (lo32(i), hi32(i), t, level block), key = seed.
// ---------------------------------------------------------------------------
// Round keys of the Weyl schedule (key + r * (0x9E3779B9, 0xBB67AE85)), computed
// on the host and passed in the kernel parameters, so every XOR reads its key
// from the constant bank.
using PhiloxKeys = PhiloxRoundKeys;

__device__ __forceinline__ uint4 philox4x32_10(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3,
                                               const PhiloxKeys& k) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint32_t lo0 = 0xD2511F53u * c0;
    const uint32_t hi0 = __umulhi(0xD2511F53u, c0);
    const uint32_t lo1 = 0xCD9E8D57u * c2;
    const uint32_t hi1 = __umulhi(0xCD9E8D57u, c2);
    c0 = hi1 ^ c1 ^ k.k0[r];
    c1 = lo1;
    c2 = hi0 ^ c3 ^ k.k1[r];
    c3 = lo0;
  }
  return make_uint4(c0, c1, c2, c3);
}

__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ float fast_log2(float x) {
  float y;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ float fast_rcp(float x) {
  float y;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Two weights at a time: packed fp32 pair arithmetic (f32x2 instructions, one
// issue for two correctly rounded operations).
__device__ __forceinline__ float2 f2(float a) { return make_float2(a, a); }
__device__ __forceinline__ float2 add2(float2 a, float2 b) { return __fadd2_rn(a, b); }
__device__ __forceinline__ float2 mul2(float2 a, float2 b) { return __fmul2_rn(a, b); }
__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c) { return __ffma2_rn(a, b, c); }
__device__ __forceinline__ float2 neg2(float2 a) { return make_float2(-a.x, -a.y); }
__device__ __forceinline__ float2 rcp2(float2 a) { return make_float2(fast_rcp(a.x), fast_rcp(a.y)); }
__device__ __forceinline__ float2 exp2_2(float2 a) { return make_float2(fast_exp2(a.x), fast_exp2(a.y)); }

// log2(u) for u in [2^-24, 1 - 2^-24], accurate to a few ulp in relative terms
// even as u -> 1 (where log2 u -> 0).  Branch-free range reduction u = 2^e m
// with m in [sqrt(1/2), sqrt(2)): subtracting the bit pattern of sqrt(1/2) from
// the bits of u moves the exponent boundary to sqrt(2) (the integer-offset
// reduction of fdlibm-style logf).  Then log2 m = (2 / ln 2) atanh(y),
// y = (m - 1)/(m + 1), by the odd series 2(y + y^3/3 + y^5/5 + ...)
// (Abramowitz & Stegun 4.1.27); |y| <= 0.1716, so terms through y^9 leave a
// relative remainder below 2e-9.
// Arithmetic right shift by 23 of one 32-bit lane.  Written in PTX: with
// nvcc 13.0 for sm_103a the C++ form of the two lanes' shifts below was
// combined into one operation on the register pair that corrupted lane x.
__device__ __forceinline__ int sar23(uint32_t x) {
  int r;
  asm("shr.s32 %0, %1, 23;" : "=r"(r) : "r"(x));
  return r;
}

__device__ __forceinline__ float2 log2_unit2(float2 u) {
  constexpr float c1 = 2.8853900817779268f;  // 2 / ln 2
  constexpr float c3 = c1 / 3.0f, c5 = c1 / 5.0f, c7 = c1 / 7.0f, c9 = c1 / 9.0f;
  const uint32_t b0 = __float_as_uint(u.x), b1 = __float_as_uint(u.y);
  const int e0 = sar23(b0 - 0x3F3504F3u);
  const int e1 = sar23(b1 - 0x3F3504F3u);
  const float2 m = make_float2(__uint_as_float(b0 + static_cast<uint32_t>(e0) * 0xFF800000u),
                               __uint_as_float(b1 + static_cast<uint32_t>(e1) * 0xFF800000u));
  const float2 y = mul2(add2(m, f2(-1.0f)), rcp2(add2(m, f2(1.0f))));
  const float2 y2 = mul2(y, y);
  float2 poly = fma2(y2, f2(c9), f2(c7));
  poly = fma2(y2, poly, f2(c5));
  poly = fma2(y2, poly, f2(c3));
  poly = fma2(y2, poly, f2(c1));
  return fma2(y, poly, make_float2(static_cast<float>(e0), static_cast<float>(e1)));
}

// The Gumbel draw in log2 units, up to a constant common to every level:
//   g = -ln(-ln u) = -ln 2 * [log2(-log2 u) + log2(ln 2)],
// so g * log2(e) = -log2(-log2 u) - log2(ln 2).  The softmax over levels is
// invariant to a shift shared by all levels, so the kernels use
//   h = -log2(-log2 u),  z'_k = kappa log2(e) l_k + h_k,  p = softmax(z'/tau in log2 units),
// which equals softmax((kappa l + g)/tau) (Alg. 1).  u = (x mod 2^23 + 1/2) 2^-23 is
// built exactly from the low 23 bits of the Philox word.  Two words -> two draws.
__device__ __forceinline__ float2 gumbel_log2_2(uint32_t x0, uint32_t x1) {
  const float2 one_plus = make_float2(__uint_as_float(0x3F800000u | (x0 & 0x007FFFFFu)),
                                      __uint_as_float(0x3F800000u | (x1 & 0x007FFFFFu)));
  const float2 u = add2(one_plus, f2(-__uint_as_float(0x3F7FFFFFu)));  // (j + 1/2) 2^-23, exact
  const float2 L = log2_unit2(u);                                      // log2 u < 0
  return make_float2(-fast_log2(-L.x), -fast_log2(-L.y));
}

// Noise of weights i0 (even) and i0 + 1 for every level (one Philox call per
// weight and block of four levels).
template <int K>
__device__ __forceinline__ void draw_noise2(const PhiloxKeys& keys, uint32_t t, uint64_t i0,
                                            int noise, float2 (&h)[K]) {
  if (!noise) {
#pragma unroll
    for (int k = 0; k < K; ++k) h[k] = f2(0.0f);
    return;
  }
#pragma unroll
  for (int blk = 0; blk < (K + 3) / 4; ++blk) {
    const uint32_t lo = static_cast<uint32_t>(i0), hi = static_cast<uint32_t>(i0 >> 32);
    const uint4 a = philox4x32_10(lo, hi, t, static_cast<uint32_t>(blk), keys);
    const uint4 b = philox4x32_10(lo + 1u, hi, t, static_cast<uint32_t>(blk), keys);
    const uint32_t wa[4] = {a.x, a.y, a.z, a.w}, wb[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (4 * blk + j < K) h[4 * blk + j] = gumbel_log2_2(wa[j], wb[j]);
  }
}

// Level value of every logit for two weights.  Full parameterisation: the grid
// (the same for every weight).  Local shift (§3.2): logit d of a weight with
// initial index j0 stands for grid[clip(j0 + d - 2, 0, nlev - 1)]; the grid is
// read from a shared-memory copy (8 words in 8 banks: no conflicts).
// The full grid is kept as scalars (no per-pair copy held in registers).
template <int K, bool kShift>
struct Levels2;

template <int K>
struct Levels2<K, false> {
  float q[K];
  __device__ __forceinline__ Levels2(const float (&q_)[kMaxLevels], const float*, int, uint32_t,
                                     uint32_t) {
#pragma unroll
    for (int k = 0; k < K; ++k) q[k] = q_[k];
  }
  __device__ __forceinline__ float x(int k) const { return q[k]; }
  __device__ __forceinline__ float y(int k) const { return q[k]; }
  __device__ __forceinline__ float2 operator[](int k) const { return f2(q[k]); }
};

template <int K>
struct Levels2<K, true> {
  float2 v[K];
  __device__ __forceinline__ Levels2(const float (&)[kMaxLevels], const float* sgrid, int nlev,
                                     uint32_t ja, uint32_t jb) {
#pragma unroll
    for (int d = 0; d < K; ++d) {
      const int ia = min(max(static_cast<int>(ja) + d - 2, 0), nlev - 1);
      const int ib = min(max(static_cast<int>(jb) + d - 2, 0), nlev - 1);
      v[d] = make_float2(sgrid[ia], sgrid[ib]);
    }
  }
  __device__ __forceinline__ float x(int k) const { return v[k].x; }
  __device__ __forceinline__ float y(int k) const { return v[k].y; }
  __device__ __forceinline__ float2 operator[](int k) const { return v[k]; }
};

// Tempered softmax over the levels and the soft value (Alg. 1), two weights:
//   p_k = exp((kappa l_k + g_k)/tau) / sum_j (...),  w~ = sum_k p_k q_k,
// evaluated as p_k = 2^((z'_k - z'_max)/tau) / sum_j 2^(...) with z' from the
// draw above (kappa_log2 = kappa log2 e).  w~ is carried as q_m + delta,
// delta = sum_j p_j (q_j - q_m), m = argmax z', so q_k - w~ = (q_k - q_m) - delta
// keeps full relative accuracy when p is nearly one-hot.
template <int K>
struct Soft2 {
  float2 p[K];
  float2 qm;
  float2 delta;
};

template <int K, class Lv>
__device__ __forceinline__ void relax2(const float2 (&l)[K], const float2 (&h)[K],
                                       float kappa_log2, float inv_tau, const Lv& qv,
                                       Soft2<K>& s) {
  float2 z[K];
  float zx = -INFINITY, zy = -INFINITY, qx = qv.x(0), qy = qv.y(0);
#pragma unroll
  for (int k = 0; k < K; ++k) {
    z[k] = fma2(f2(kappa_log2), l[k], h[k]);
    if (z[k].x > zx) {
      zx = z[k].x;
      qx = qv.x(k);
    }
    if (z[k].y > zy) {
      zy = z[k].y;
      qy = qv.y(k);
    }
  }
  const float2 qm = make_float2(qx, qy);
  const float2 off = mul2(make_float2(zx, zy), f2(-inv_tau));
  float2 sum = f2(0.0f), delta = f2(0.0f);
#pragma unroll
  for (int k = 0; k < K; ++k) {
    s.p[k] = exp2_2(fma2(z[k], f2(inv_tau), off));
    sum = add2(sum, s.p[k]);
    delta = fma2(s.p[k], add2(qv[k], neg2(qm)), delta);
  }
  const float2 inv = rcp2(sum);
#pragma unroll
  for (int k = 0; k < K; ++k) s.p[k] = mul2(s.p[k], inv);
  s.qm = qm;
  s.delta = mul2(delta, inv);
}

// Soft value only (forward), two weights:
//   w~ = sum_k 2^((z'_k - z'_max)/tau) q_k / sum_k 2^(...).
template <int K, class Lv>
__device__ __forceinline__ float2 soft_value2(const float2 (&l)[K], const float2 (&h)[K],
                                              float kappa_log2, float inv_tau, const Lv& qv) {
  float2 z[K];
  float zx = -INFINITY, zy = -INFINITY;
#pragma unroll
  for (int k = 0; k < K; ++k) {
    z[k] = fma2(f2(kappa_log2), l[k], h[k]);
    zx = fmaxf(zx, z[k].x);
    zy = fmaxf(zy, z[k].y);
  }
  const float2 off = mul2(make_float2(zx, zy), f2(-inv_tau));
  float2 sum = f2(0.0f), num = f2(0.0f);
#pragma unroll
  for (int k = 0; k < K; ++k) {
    const float2 e = exp2_2(fma2(z[k], f2(inv_tau), off));
    sum = add2(sum, e);
    num = fma2(e, qv[k], num);
  }
  return mul2(num, rcp2(sum));
}

__device__ __forceinline__ void load_w4(const void* W, int64_t q, int bf16, float (&w)[4]) {
  if (bf16) {
    const uint2 raw = __ldg(reinterpret_cast<const uint2*>(W) + q);
    const __nv_bfloat162 a = *reinterpret_cast<const __nv_bfloat162*>(&raw.x);
    const __nv_bfloat162 b = *reinterpret_cast<const __nv_bfloat162*>(&raw.y);
    const float2 fa = __bfloat1622float2(a), fb = __bfloat1622float2(b);
    w[0] = fa.x; w[1] = fa.y; w[2] = fb.x; w[3] = fb.y;
  } else {
    const float4 v = __ldg(reinterpret_cast<const float4*>(W) + q);
    w[0] = v.x; w[1] = v.y; w[2] = v.z; w[3] = v.w;
  }
}

// Rounds D to its storage precision in place and stores it.
__device__ __forceinline__ void store_d4(void* D, int64_t q, int bf16, float (&d)[4]) {
  if (bf16) {
    const __nv_bfloat162 a = __floats2bfloat162_rn(d[0], d[1]);
    const __nv_bfloat162 b = __floats2bfloat162_rn(d[2], d[3]);
    const float2 fa = __bfloat1622float2(a), fb = __bfloat1622float2(b);
    d[0] = fa.x; d[1] = fa.y; d[2] = fb.x; d[3] = fb.y;
    uint2 raw;
    raw.x = *reinterpret_cast<const uint32_t*>(&a);
    raw.y = *reinterpret_cast<const uint32_t*>(&b);
    reinterpret_cast<uint2*>(D)[q] = raw;
  } else {
    reinterpret_cast<float4*>(D)[q] = make_float4(d[0], d[1], d[2], d[3]);
  }
}

__device__ __forceinline__ float round_d(float d, int bf16) {
  return bf16 ? __bfloat162float(__float2bfloat16_rn(d)) : d;
}

// lr * sign(c) with sign(0) = 0.
__device__ __forceinline__ float lr_sign(float lr, float c) {
  return c != 0.0f ? copysignf(lr, c) : 0.0f;
}

__device__ __forceinline__ float group_sum(float v, int seg) {
  for (int off = 1; off < seg; off <<= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}

__device__ __forceinline__ void load_grid(const EwParams& P, float (&q)[kMaxLevels]) {
#pragma unroll
  for (int k = 0; k < kMaxLevels; ++k) q[k] = P.grid[k];
}

// Block-wide shared copy of the grid (local shift reads it with per-lane indices).
__device__ __forceinline__ void fill_shared_grid(const EwParams& P, float* sgrid) {
  if (threadIdx.x < kMaxLevels) sgrid[threadIdx.x] = P.grid[threadIdx.x];
  __syncthreads();
}

__device__ __forceinline__ uint32_t load_j0(const EwParams& P, int64_t q) {
  return reinterpret_cast<const uint32_t*>(P.j0)[q];
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
  if (is_last && threadIdx.x == 0) {
    __threadfence();
    double s = 0.0;
    for (unsigned int b = 0; b < gridDim.x; ++b) s += __ldcg(P.loss_partials + b);
    if (P.loss_out) *P.loss_out = static_cast<float>(s);
    P.flags->blocks_done = 0u;
  }
}

// ---------------------------------------------------------------------------
// Relaxation policies: how a pair of weights' logits and noise become their
// soft values w~ and how dw~/dl flows back.  One fused kernel skeleton serves
// all of them.
//   L             logits per weight (planes of the logit tensors)
//   noise(...)    the step's draws for the pair, in log2 units
//   relax(...)    w~ of the pair; keeps what dsoft() needs
//   dsoft(k)      dw~/dl_k divided by kappa/tau
//   value(...)    w~ only (forward)
// ---------------------------------------------------------------------------
// Categorical GS over the K grid levels (Alg. 1), or over 5 local shifts.
template <int K, bool kShift>
struct CatRelax {
  static constexpr int L = K;
  Levels2<K, kShift> qv;
  Soft2<K> sm;
  __device__ __forceinline__ CatRelax(const float (&q)[kMaxLevels], const float* sgrid, int nlev,
                                      uint32_t ja, uint32_t jb)
      : qv(q, sgrid, nlev, ja, jb) {}
  __device__ static __forceinline__ void noise(const PhiloxKeys& keys, uint32_t t, uint64_t i0,
                                               int on, float2 (&h)[L]) {
    draw_noise2<K>(keys, t, i0, on, h);
  }
  __device__ __forceinline__ float2 relax(const float2 (&l)[L], const float2 (&h)[L],
                                          float kappa_log2, float inv_tau) {
    relax2<K>(l, h, kappa_log2, inv_tau, qv, sm);
    return add2(sm.qm, sm.delta);
  }
  // softmax Jacobian (App. B): dw~/dl_k = (kappa/tau) p_k (q_k - w~)
  __device__ __forceinline__ float2 dsoft(int k) const {
    return mul2(sm.p[k], add2(add2(qv[k], neg2(sm.qm)), neg2(sm.delta)));
  }
  __device__ __forceinline__ float2 value(const float2 (&l)[L], const float2 (&h)[L],
                                          float kappa_log2, float inv_tau) const {
    return soft_value2<K>(l, h, kappa_log2, inv_tau, qv);
  }
};

// Logistic(0, 1) draws in log2 units, log2(u / (1 - u)), for weights i0 (even)
// and i0 + 1, which share one Philox block (counter of i0, block 0): words 0
// and 1 are the mask and sign draws of i0, words 2 and 3 those of i0 + 1.  A
// binary GS over tied logits (-l, l) sees only the difference g1 - g0 of its
// two Gumbel draws, whose law this is.  u and 1 - u are both exact: the
// complemented 23 bits give 1 - u.
__device__ __forceinline__ void draw_logistic2(const PhiloxKeys& keys, uint32_t t, uint64_t i0,
                                               int on, float2 (&h)[2]) {
  if (!on) {
    h[0] = h[1] = f2(0.0f);
    return;
  }
  const uint4 a = philox4x32_10(static_cast<uint32_t>(i0), static_cast<uint32_t>(i0 >> 32), t, 0u,
                                keys);
  const float half = __uint_as_float(0x3F7FFFFFu);  // 1 - 2^-24
  auto unit = [&](uint32_t x) { return __uint_as_float(0x3F800000u | (x & 0x007FFFFFu)) - half; };
  // u / (1 - u) for (mask, mask) and (sign, sign) of the two weights
  const float2 um = make_float2(unit(a.x), unit(a.z)), vm = make_float2(unit(~a.x), unit(~a.z));
  const float2 ub = make_float2(unit(a.y), unit(a.w)), vb = make_float2(unit(~a.y), unit(~a.w));
  h[0] = log2_unit2(mul2(um, rcp2(vm)));
  h[1] = log2_unit2(mul2(ub, rcp2(vb)));
}

// Ternary mask x sign (§3.1, Alg. 2): w~ = a m~ b~ on the grid {-a, 0, a}, with
// m~ = GS({0,1}, (-l_m, l_m)) and b~ = GS({-1,1}, (-l_b, l_b)); each binary GS
// is a sigmoid of the noisy logit 2l (§3 notation paragraph):
//   y = (2 kappa log2(e) l + log2(u/(1-u))) / tau,  p1 = 1 / (1 + 2^-y).
// With e = 2^-|y| and r = 1/(1+e): the larger of p0, p1 is r, the smaller e r
// (no overflow for any y), p0 p1 = e r^2, p1 - p0 = sign(y) (1 - e) r.
// dm~/dl_m = 2 (kappa/tau) p0 p1, db~/dl_b = 4 (kappa/tau) p0 p1.
struct MaskSignRelax {
  static constexpr int L = 2;
  float a;
  float2 mt, bt, gm, gb;
  __device__ __forceinline__ MaskSignRelax(const float (&q)[kMaxLevels], const float*, int, uint32_t,
                                           uint32_t)
      : a(q[2]) {}
  __device__ static __forceinline__ void noise(const PhiloxKeys& keys, uint32_t t, uint64_t i0,
                                               int on, float2 (&h)[L]) {
    draw_logistic2(keys, t, i0, on, h);
  }
  struct Bin {
    float2 hi, lo, y;   // max(p0,p1), min(p0,p1), y
  };
  __device__ static __forceinline__ Bin binary(float2 l, float2 h, float kappa_log2, float inv_tau) {
    Bin b;
    b.y = mul2(fma2(f2(2.0f * kappa_log2), l, h), f2(inv_tau));
    const float2 e = exp2_2(make_float2(-fabsf(b.y.x), -fabsf(b.y.y)));
    b.hi = rcp2(add2(e, f2(1.0f)));
    b.lo = mul2(e, b.hi);
    return b;
  }
  __device__ static __forceinline__ float2 p1(const Bin& b) {
    return make_float2(b.y.x >= 0.0f ? b.hi.x : b.lo.x, b.y.y >= 0.0f ? b.hi.y : b.lo.y);
  }
  __device__ static __forceinline__ float2 pm(const Bin& b) {   // p1 - p0
    const float2 d = add2(b.hi, neg2(b.lo));
    return make_float2(copysignf(d.x, b.y.x), copysignf(d.y, b.y.y));
  }
  __device__ __forceinline__ float2 relax(const float2 (&l)[L], const float2 (&h)[L],
                                          float kappa_log2, float inv_tau) {
    const Bin m = binary(l[0], h[0], kappa_log2, inv_tau);
    const Bin b = binary(l[1], h[1], kappa_log2, inv_tau);
    mt = p1(m);
    bt = pm(b);
    gm = mul2(f2(2.0f), mul2(m.hi, m.lo));
    gb = mul2(f2(4.0f), mul2(b.hi, b.lo));
    return mul2(f2(a), mul2(mt, bt));
  }
  __device__ __forceinline__ float2 dsoft(int k) const {
    return k == 0 ? mul2(f2(a), mul2(bt, gm)) : mul2(f2(a), mul2(mt, gb));
  }
  __device__ __forceinline__ float2 value(const float2 (&l)[L], const float2 (&h)[L],
                                          float kappa_log2, float inv_tau) const {
    const Bin m = binary(l[0], h[0], kappa_log2, inv_tau);
    const Bin b = binary(l[1], h[1], kappa_log2, inv_tau);
    return mul2(f2(a), mul2(p1(m), pm(b)));
  }
};

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

template <class Rx, bool kExport, bool kShift, bool kAcc>
__global__ void __launch_bounds__(kEwThreads, BwdOcc<Rx::L>::value) k_backward(const EwParams P) {
  constexpr int K = Rx::L;
  float q[kMaxLevels];
  load_grid(P, q);
  __shared__ float sgrid[kMaxLevels];
  if (kShift) fill_shared_grid(P, sgrid);
  const PhiloxKeys& keys = P.keys;
  const int lane = threadIdx.x & 31;
  const int seg = P.group >> 2;  // lanes per scale group
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  float2 loss2 = f2(0.0f);

  for (int64_t base = static_cast<int64_t>(blockIdx.x) * blockDim.x + (threadIdx.x & ~31);
       base < P.nq; base += stride) {
    const int64_t qi = base + lane;
    const bool active = qi < P.nq;
    const int64_t qc = active ? qi : 0;
    // Lanes past the end (only in the last warp) read quad 0 and take G = 0, so
    // every value stays finite and their loss and scale-gradient terms vanish;
    // nothing is stored for them.  A scale group is never split across active
    // and inactive lanes.
    float l[K][4], m[K][4];
    float w[4];
    float s, ms = 0.0f;
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
    float4 gv = __ldcs(reinterpret_cast<const float4*>(P.G) + qc);
    if (!active) gv = make_float4(0.f, 0.f, 0.f, 0.f);
    load_w4(P.W, qc, P.w_bf16, w);
    s = __ldg(P.scales + gidx);
    if (!kExport && !P.scales_frozen) ms = __ldg(P.m_scales + gidx);
    const float2 Gq[2] = {make_float2(gv.x, gv.y), make_float2(gv.z, gv.w)};
    const uint32_t j4 = kShift ? load_j0(P, qc) : 0u;
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
  reduce_loss(loss2.x + loss2.y, P);
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


template <class T>
struct Tag {
  using type = T;
};

// The relaxation policy of a layer: categorical over K levels, local shift
// (K = 5 only) or mask x sign (2 logits).
template <class F>
cudaError_t with_relax(int K, int mode, F&& f) {
  switch (mode) {
    case GSQ_PARAM_SHIFT5:
      if (K != 5) return cudaErrorInvalidValue;
      f(Tag<CatRelax<5, true>>{}, std::true_type{});
      return cudaSuccess;
    case GSQ_PARAM_MASK_SIGN:
      if (K != 2) return cudaErrorInvalidValue;
      f(Tag<MaskSignRelax>{}, std::false_type{});
      return cudaSuccess;
    default:
      break;
  }
  switch (K) {
    case 2: f(Tag<CatRelax<2, false>>{}, std::false_type{}); break;
    case 3: f(Tag<CatRelax<3, false>>{}, std::false_type{}); break;
    case 4: f(Tag<CatRelax<4, false>>{}, std::false_type{}); break;
    case 5: f(Tag<CatRelax<5, false>>{}, std::false_type{}); break;
    case 6: f(Tag<CatRelax<6, false>>{}, std::false_type{}); break;
    case 7: f(Tag<CatRelax<7, false>>{}, std::false_type{}); break;
    case 8: f(Tag<CatRelax<8, false>>{}, std::false_type{}); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaSuccess;
}

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
