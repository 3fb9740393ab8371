// Device code shared by the forward and backward elementwise kernels:
// counter-based Gumbel / logistic noise (Philox4x32-10), packed fp32 pair
// arithmetic, the tempered softmax of a categorical relaxation and the binary
// mask x sign relaxation, with their Jacobians (App. B).  Internal linkage:
// every translation unit that includes it gets its own copy.
#pragma once

#include <cuda_bf16.h>

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
// (Abramowitz & Stegun 4.1.27); |y| <= 0.1716, so terms through y^7 leave a
// relative remainder below y^8/9 = 8.3e-8 (under 1.5 ulp of fp32).
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
  constexpr float c3 = c1 / 3.0f, c5 = c1 / 5.0f, c7 = c1 / 7.0f;
  const uint32_t b0 = __float_as_uint(u.x), b1 = __float_as_uint(u.y);
  const int e0 = sar23(b0 - 0x3F3504F3u);
  const int e1 = sar23(b1 - 0x3F3504F3u);
  const float2 m = make_float2(__uint_as_float(b0 + static_cast<uint32_t>(e0) * 0xFF800000u),
                               __uint_as_float(b1 + static_cast<uint32_t>(e1) * 0xFF800000u));
  const float2 y = mul2(add2(m, f2(-1.0f)), rcp2(add2(m, f2(1.0f))));
  const float2 y2 = mul2(y, y);
  float2 poly = fma2(y2, f2(c7), f2(c5));
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

// Noise of two weights with flat indices ia and ib for every level: each
// weight's draw comes from its own counter (lo32(i), hi32(i), t, level block),
// one Philox call per weight and block of four levels.
template <int K>
__device__ __forceinline__ void draw_noise_pair(const PhiloxKeys& keys, uint32_t t, uint64_t ia,
                                                uint64_t ib, int noise, float2 (&h)[K]) {
  if (!noise) {
#pragma unroll
    for (int k = 0; k < K; ++k) h[k] = f2(0.0f);
    return;
  }
#pragma unroll
  for (int blk = 0; blk < (K + 3) / 4; ++blk) {
    const uint4 a = philox4x32_10(static_cast<uint32_t>(ia), static_cast<uint32_t>(ia >> 32), t,
                                  static_cast<uint32_t>(blk), keys);
    const uint4 b = philox4x32_10(static_cast<uint32_t>(ib), static_cast<uint32_t>(ib >> 32), t,
                                  static_cast<uint32_t>(blk), keys);
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
// draw above (kappa_log2 = kappa log2 e); the numerators and 1/sum are kept
// apart (the backward folds 1/sum into its per-weight factor).  w~ is carried as q_m + delta,
// delta = sum_j p_j (q_j - q_m), m = argmax z', so q_k - w~ = (q_k - q_m) - delta
// keeps full relative accuracy when p is nearly one-hot.
template <int K>
struct Soft2 {
  float2 p[K];   // 2^((z'_k - z'_max)/tau): p_k before the division by their sum
  float2 inv;    // 1 / sum
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
  s.inv = inv;
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

__device__ __forceinline__ float round_d(float d, int bf16) {
  return bf16 ? __bfloat162float(__float2bfloat16_rn(d)) : d;
}

// lr * sign(c) with sign(0) = 0.
__device__ __forceinline__ float lr_sign(float lr, float c) {
  return c != 0.0f ? copysignf(lr, c) : 0.0f;
}

// ---------------------------------------------------------------------------
// Relaxation policies: how a pair of weights' logits and noise become their
// soft values w~ and how dw~/dl flows back.  One fused kernel skeleton serves
// all of them.
//   L             logits per weight (planes of the logit tensors)
//   noise(...)    the step's draws for the pair, in log2 units
//   relax(...)    w~ of the pair; keeps what dsoft() needs
//   dsoft(k)      dw~/dl_k divided by kappa/tau, times 1/dscale()
//   kScaled       whether dscale() is not 1
//   value(...)    w~ only (forward)
// ---------------------------------------------------------------------------
// Categorical GS over the K grid levels (Alg. 1), or over 5 local shifts.
template <int K, bool kShift>
struct CatRelax {
  static constexpr int L = K;
  static constexpr bool kScaled = true;
  Levels2<K, kShift> qv;
  Soft2<K> sm;
  __device__ __forceinline__ CatRelax(const float (&q)[kMaxLevels], const float* sgrid, int nlev,
                                      uint32_t ja, uint32_t jb)
      : qv(q, sgrid, nlev, ja, jb) {}
  // weights i0 (even) and i0 + 1
  __device__ static __forceinline__ void noise(const PhiloxKeys& keys, uint32_t t, uint64_t i0,
                                               int on, float2 (&h)[L]) {
    draw_noise_pair<K>(keys, t, i0, i0 + 1, on, h);
  }
  __device__ __forceinline__ float2 relax(const float2 (&l)[L], const float2 (&h)[L],
                                          float kappa_log2, float inv_tau) {
    relax2<K>(l, h, kappa_log2, inv_tau, qv, sm);
    return add2(sm.qm, sm.delta);
  }
  // softmax Jacobian (App. B): dw~/dl_k = (kappa/tau) p_k (q_k - w~), here with the
  // numerator of p_k; dscale() is the 1/sum that completes it
  __device__ __forceinline__ float2 dsoft(int k) const {
    return mul2(sm.p[k], add2(add2(qv[k], neg2(sm.qm)), neg2(sm.delta)));
  }
  __device__ __forceinline__ float2 dscale() const { return sm.inv; }
  __device__ __forceinline__ float2 value(const float2 (&l)[L], const float2 (&h)[L],
                                          float kappa_log2, float inv_tau) const {
    return soft_value2<K>(l, h, kappa_log2, inv_tau, qv);
  }
};

// h[0] = log2(u/(1-u)) of the mask words (ma, mb), h[1] of the sign words (sa, sb),
// u = (x mod 2^23 + 1/2) 2^-23 from the low 23 bits of each word.
__device__ __forceinline__ void logistic_from_words2(uint32_t ma, uint32_t mb, uint32_t sa,
                                                     uint32_t sb, float2 (&h)[2]) {
  const float half = __uint_as_float(0x3F7FFFFFu);  // 1 - 2^-24
  auto unit = [&](uint32_t x) { return __uint_as_float(0x3F800000u | (x & 0x007FFFFFu)) - half; };
  const float2 um = make_float2(unit(ma), unit(mb)), vm = make_float2(unit(~ma), unit(~mb));
  const float2 ub = make_float2(unit(sa), unit(sb)), vb = make_float2(unit(~sa), unit(~sb));
  h[0] = log2_unit2(mul2(um, rcp2(vm)));
  h[1] = log2_unit2(mul2(ub, rcp2(vb)));
}

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
  logistic_from_words2(a.x, a.z, a.y, a.w, h);
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
  static constexpr bool kScaled = false;
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
  __device__ __forceinline__ float2 dscale() const { return f2(1.0f); }
  __device__ __forceinline__ float2 value(const float2 (&l)[L], const float2 (&h)[L],
                                          float kappa_log2, float inv_tau) const {
    const Bin m = binary(l[0], h[0], kappa_log2, inv_tau);
    const Bin b = binary(l[1], h[1], kappa_log2, inv_tau);
    return mul2(f2(a), mul2(p1(m), pm(b)));
  }
};

// ---- quad access: one thread owns 4 consecutive weights (quad q = i / 4) ----
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

__device__ __forceinline__ float group_sum(float v, int seg) {
  for (int off = 1; off < seg; off <<= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}

__device__ __forceinline__ uint32_t load_j0(const EwParams& P, int64_t q) {
  return reinterpret_cast<const uint32_t*>(P.j0)[q];
}

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

}  // namespace
}  // namespace gsq
