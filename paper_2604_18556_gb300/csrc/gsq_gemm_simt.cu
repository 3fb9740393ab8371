// CUDA-core GEMM for the fp32 validation path of the loss contraction
// (G = 2 D H_sym, Eq. 1 with a linear layer) and for forming H = X^T X from
// calibration tokens at init; plus the symmetrisation / precision conversion of
// H.  Not the performance path: the bf16 contraction runs on the tensor cores.
#include <cuda_bf16.h>

#include "gsq_internal.h"

namespace gsq {
namespace {

constexpr int BM = 64, BN = 64, BK = 16, TM = 4, TN = 4;

template <bool kBf16>
__device__ __forceinline__ float ld_in(const void* p, int64_t idx) {
  if (kBf16) return __bfloat162float(reinterpret_cast<const __nv_bfloat16*>(p)[idx]);
  return reinterpret_cast<const float*>(p)[idx];
}

// C[b][m][n] = alpha * sum_k A[b][m*sam + k*sak] * B[b][k*sbk + n*sbn], fp32 accumulate.
template <bool kBf16>
__global__ void __launch_bounds__(256) k_simt_gemm(const SimtGemm g) {
  __shared__ float As[BK][BM + 4];
  __shared__ float Bs[BK][BN + 4];
  const int b = blockIdx.z;
  const int m0 = blockIdx.y * BM, n0 = blockIdx.x * BN;
  const int tid = threadIdx.x;
  const int tx = tid % (BN / TN), ty = tid / (BN / TN);
  const char* Ab = reinterpret_cast<const char*>(g.A) + b * g.sab * (kBf16 ? 2 : 4);
  const char* Bb = reinterpret_cast<const char*>(g.B) + b * g.sbb * (kBf16 ? 2 : 4);
  float acc[TM][TN];
#pragma unroll
  for (int i = 0; i < TM; ++i)
#pragma unroll
    for (int j = 0; j < TN; ++j) acc[i][j] = 0.0f;
  for (int k0 = 0; k0 < g.Kd; k0 += BK) {
    for (int e = tid; e < BM * BK; e += 256) {
      const int mm = e / BK, kk = e % BK;
      const int gm = m0 + mm, gk = k0 + kk;
      As[kk][mm] = (gm < g.M && gk < g.Kd) ? ld_in<kBf16>(Ab, gm * g.sam + gk * g.sak) : 0.0f;
    }
    for (int e = tid; e < BN * BK; e += 256) {
      const int kk = e / BN, nn = e % BN;
      const int gk = k0 + kk, gn = n0 + nn;
      Bs[kk][nn] = (gk < g.Kd && gn < g.N) ? ld_in<kBf16>(Bb, gk * g.sbk + gn * g.sbn) : 0.0f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < BK; ++kk) {
      float a[TM], bb[TN];
#pragma unroll
      for (int i = 0; i < TM; ++i) a[i] = As[kk][ty * TM + i];
#pragma unroll
      for (int j = 0; j < TN; ++j) bb[j] = Bs[kk][tx * TN + j];
#pragma unroll
      for (int i = 0; i < TM; ++i)
#pragma unroll
        for (int j = 0; j < TN; ++j) acc[i][j] = fmaf(a[i], bb[j], acc[i][j]);
    }
    __syncthreads();
  }
  float* Cb = g.C + b * g.scb;
#pragma unroll
  for (int i = 0; i < TM; ++i) {
    const int gm = m0 + ty * TM + i;
    if (gm >= g.M) continue;
#pragma unroll
    for (int j = 0; j < TN; ++j) {
      const int gn = n0 + tx * TN + j;
      if (gn < g.N) Cb[static_cast<int64_t>(gm) * g.ldc + gn] = g.alpha * acc[i][j];
    }
  }
}

// out[e] = (H[e] + H[e]^T) / 2 in bf16 or fp32, through a 32x32 shared tile.
template <bool kBf16Out>
__global__ void k_symmetrize(const float* H, void* out, int C) {
  __shared__ float t[32][33];
  const int e = blockIdx.z;
  const int64_t base = static_cast<int64_t>(e) * C * C;
  const int i0 = blockIdx.y * 32, j0 = blockIdx.x * 32;
  const int tx = threadIdx.x, ty = threadIdx.y;  // 32 x 8
  for (int r = ty; r < 32; r += 8) {
    const int i = j0 + r, j = i0 + tx;  // transposed tile: H[j0 + r][i0 + tx]
    t[r][tx] = (i < C && j < C) ? H[base + static_cast<int64_t>(i) * C + j] : 0.0f;
  }
  __syncthreads();
  for (int r = ty; r < 32; r += 8) {
    const int i = i0 + r, j = j0 + tx;
    if (i < C && j < C) {
      const float v = (H[base + static_cast<int64_t>(i) * C + j] + t[tx][r]) * 0.5f;
      if (kBf16Out)
        reinterpret_cast<__nv_bfloat16*>(out)[base + static_cast<int64_t>(i) * C + j] =
            __float2bfloat16_rn(v);
      else
        reinterpret_cast<float*>(out)[base + static_cast<int64_t>(i) * C + j] = v;
    }
  }
}

// H[e][i][j] = H[e][j][i] for i > j (bf16, C even): the lower triangle from the upper
// one.  One block per 64 x 64 destination tile on or below the diagonal (blocks
// enumerated over the triangle): the source tile above the diagonal is read with
// 4-byte loads of two columns into shared memory, the destination written with 4-byte
// stores of two columns.  A block reads only the upper triangle and writes only the
// lower one (a diagonal tile reads all of itself before writing), so blocks never race.
__global__ void __launch_bounds__(256) k_mirror_upper_bf16(__nv_bfloat16* H, int C) {
  const int x = blockIdx.x;
  int bi = static_cast<int>((sqrtf(8.0f * static_cast<float>(x) + 1.0f) - 1.0f) * 0.5f);
  while ((bi + 1) * (bi + 2) / 2 <= x) ++bi;
  while (bi * (bi + 1) / 2 > x) --bi;
  const int bj = x - bi * (bi + 1) / 2;  // destination tile: rows bi, columns bj <= bi
  __shared__ __align__(4) __nv_bfloat16 t[64][66];
  __nv_bfloat16* He = H + static_cast<int64_t>(blockIdx.y) * C * C;
  const int i0 = bi * 64, j0 = bj * 64;
  for (int k = threadIdx.x; k < 64 * 32; k += 256) {  // source rows j0.., columns i0..
    const int r = k >> 5, c = (k & 31) * 2;
    const int gi = j0 + r, gj = i0 + c;
    if (gi < C && gj < C)
      *reinterpret_cast<uint32_t*>(&t[r][c]) =
          *reinterpret_cast<const uint32_t*>(He + static_cast<int64_t>(gi) * C + gj);
  }
  __syncthreads();
  for (int k = threadIdx.x; k < 64 * 32; k += 256) {  // destination rows i0.., columns j0..
    const int r = k >> 5, c = (k & 31) * 2;
    const int gi = i0 + r, gj = j0 + c;
    if (gi >= C || gj >= C || gi <= gj) continue;
    __nv_bfloat16* dst = He + static_cast<int64_t>(gi) * C + gj;
    if (gi > gj + 1) {
      __nv_bfloat162 v;
      v.x = t[c][r];
      v.y = t[c + 1][r];
      *reinterpret_cast<__nv_bfloat162*>(dst) = v;
    } else {
      *dst = t[c][r];
    }
  }
}

// Tokens of one micro-batch to the tensor-core operands: Xb[e][t][c] and
// Xt[e][c][t] = bf16(X[e][t][c]).  One 64 x 64 tile per block of 256 threads:
// 16-byte loads along c, 8-byte stores of four bf16 to Xb, the tile through
// shared memory, then 8-byte stores of four tokens to Xt.  T and C are
// multiples of 8, so a group of four never straddles an edge.  ldt is the row
// length of Xt.
__global__ void __launch_bounds__(256) k_tokens_bf16(const float* X, __nv_bfloat16* Xb,
                                                     __nv_bfloat16* Xt, int T, int C, int ldt) {
  __shared__ __nv_bfloat16 tile[64][68];
  const int e = blockIdx.z;
  const int t0 = blockIdx.y * 64, c0 = blockIdx.x * 64;
  const int tid = threadIdx.x;
  const int q = (tid & 15) * 4, r0 = tid >> 4;  // 16 groups of four along the tile row
  const float* Xe = X + static_cast<int64_t>(e) * T * C;
  __nv_bfloat16* Xbe = Xb + static_cast<int64_t>(e) * T * C;
  __nv_bfloat16* Xte = Xt + static_cast<int64_t>(e) * C * ldt;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int r = r0 + 16 * i, t = t0 + r, c = c0 + q;
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
    if (t < T && c < C) v = __ldcs(reinterpret_cast<const float4*>(Xe + static_cast<int64_t>(t) * C + c));
    const __nv_bfloat162 lo = __floats2bfloat162_rn(v.x, v.y), hi = __floats2bfloat162_rn(v.z, v.w);
    if (t < T && c < C) {
      uint2 raw;
      raw.x = *reinterpret_cast<const uint32_t*>(&lo);
      raw.y = *reinterpret_cast<const uint32_t*>(&hi);
      *reinterpret_cast<uint2*>(Xbe + static_cast<int64_t>(t) * C + c) = raw;
    }
    *reinterpret_cast<__nv_bfloat162*>(&tile[r][q]) = lo;
    *reinterpret_cast<__nv_bfloat162*>(&tile[r][q + 2]) = hi;
  }
  __syncthreads();
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int cr = r0 + 16 * i, c = c0 + cr, t = t0 + q;
    if (c < C && t < T) {
      const __nv_bfloat162 lo = __halves2bfloat162(tile[q][cr], tile[q + 1][cr]);
      const __nv_bfloat162 hi = __halves2bfloat162(tile[q + 2][cr], tile[q + 3][cr]);
      uint2 raw;
      raw.x = *reinterpret_cast<const uint32_t*>(&lo);
      raw.y = *reinterpret_cast<const uint32_t*>(&hi);
      *reinterpret_cast<uint2*>(Xte + static_cast<int64_t>(c) * ldt + t) = raw;
    }
  }
}

// Tokens of one micro-batch to X^T alone: Xt[e][c][t] = bf16(X[e][t][c]), without
// shared memory.  Each thread reads 8 consecutive tokens x 4 channels (eight 16-byte
// loads; the 16 lanes of a half-warp cover 64 channels of one token row) and writes
// each channel's 8 tokens with one 16-byte store.  A block covers 128 tokens x 64
// channels.  T and C are multiples of 8, so a thread's tokens and channels are all
// inside or all outside the layer.
__global__ void __launch_bounds__(256) k_tokens_t_bf16(const float* X, __nv_bfloat16* Xt, int T,
                                                       int C, int ldt) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int c = blockIdx.x * 64 + (lane & 15) * 4;
  const int t0 = blockIdx.y * 128 + warp * 16 + (lane >> 4) * 8;
  if (c >= C || t0 >= T) return;
  const float* Xe = X + static_cast<int64_t>(blockIdx.z) * T * C;
  __nv_bfloat16* Xte = Xt + static_cast<int64_t>(blockIdx.z) * C * ldt;
  float4 v[8];
#pragma unroll
  for (int i = 0; i < 8; ++i)
    v[i] = __ldcs(reinterpret_cast<const float4*>(Xe + static_cast<int64_t>(t0 + i) * C + c));
  auto pack = [](float a, float b) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<const uint32_t*>(&h);
  };
  __nv_bfloat16* o = Xte + static_cast<int64_t>(c) * ldt + t0;
  *reinterpret_cast<uint4*>(o) = make_uint4(pack(v[0].x, v[1].x), pack(v[2].x, v[3].x),
                                            pack(v[4].x, v[5].x), pack(v[6].x, v[7].x));
  *reinterpret_cast<uint4*>(o + ldt) = make_uint4(pack(v[0].y, v[1].y), pack(v[2].y, v[3].y),
                                                  pack(v[4].y, v[5].y), pack(v[6].y, v[7].y));
  *reinterpret_cast<uint4*>(o + 2 * static_cast<int64_t>(ldt)) =
      make_uint4(pack(v[0].z, v[1].z), pack(v[2].z, v[3].z), pack(v[4].z, v[5].z),
                 pack(v[6].z, v[7].z));
  *reinterpret_cast<uint4*>(o + 3 * static_cast<int64_t>(ldt)) =
      make_uint4(pack(v[0].w, v[1].w), pack(v[2].w, v[3].w), pack(v[4].w, v[5].w),
                 pack(v[6].w, v[7].w));
}

// One block per canary (256 bytes = 64 words): write the pattern, or compare.
__global__ void k_canaries(uint8_t* ws, const CanaryList list, int write, DevFlags* flags) {
  const int i = blockIdx.x;
  uint32_t* c = reinterpret_cast<uint32_t*>(ws + list.off[i]);
  const uint32_t pattern = 0x5EED0000u ^ static_cast<uint32_t>(i) * 0x9E3779B1u;
  if (write) {
    c[threadIdx.x] = pattern ^ threadIdx.x;
  } else if (c[threadIdx.x] != (pattern ^ threadIdx.x)) {
    atomicCAS(&flags->error, 0u, kCanaryError | static_cast<unsigned int>(i));
  }
}

}  // namespace

cudaError_t launch_canaries(uint8_t* ws, const CanaryList& list, int write, DevFlags* flags,
                            cudaStream_t s) {
  if (list.count <= 0) return cudaSuccess;
  k_canaries<<<list.count, 64, 0, s>>>(ws, list, write, flags);
  return cudaGetLastError();
}

cudaError_t launch_tokens_bf16(const float* X, void* Xb, void* Xt, int E, int T, int C, int ldt,
                               cudaStream_t s) {
  if (E <= 0 || T <= 0 || C <= 0) return cudaSuccess;
  if (T % 8 != 0 || C % 8 != 0 || ldt % 4 != 0) return cudaErrorInvalidValue;
  if (!Xb) {  // X^T alone
    if (ldt % 8 != 0) return cudaErrorInvalidValue;  // 16-byte stores
    dim3 grid_t((C + 63) / 64, (T + 127) / 128, E);
    k_tokens_t_bf16<<<grid_t, 256, 0, s>>>(X, static_cast<__nv_bfloat16*>(Xt), T, C, ldt);
    return cudaGetLastError();
  }
  dim3 grid((C + 63) / 64, (T + 63) / 64, E);
  k_tokens_bf16<<<grid, 256, 0, s>>>(X, static_cast<__nv_bfloat16*>(Xb),
                                     static_cast<__nv_bfloat16*>(Xt), T, C, ldt);
  return cudaGetLastError();
}

cudaError_t launch_simt_gemm(const SimtGemm& g, cudaStream_t s) {
  dim3 grid((g.N + BN - 1) / BN, (g.M + BM - 1) / BM, g.batch);
  if (g.bf16_inputs)
    k_simt_gemm<true><<<grid, 256, 0, s>>>(g);
  else
    k_simt_gemm<false><<<grid, 256, 0, s>>>(g);
  return cudaGetLastError();
}

cudaError_t launch_symmetrize(const float* H, void* out, int E, int C, int out_bf16, cudaStream_t s) {
  dim3 grid((C + 31) / 32, (C + 31) / 32, E);
  dim3 block(32, 8);
  if (out_bf16)
    k_symmetrize<true><<<grid, block, 0, s>>>(H, out, C);
  else
    k_symmetrize<false><<<grid, block, 0, s>>>(H, out, C);
  return cudaGetLastError();
}

cudaError_t launch_mirror_upper_bf16(void* H, int E, int C, cudaStream_t s) {
  if (E <= 0 || C <= 0) return cudaSuccess;
  if (C % 2 != 0) return cudaErrorInvalidValue;
  const int nb = (C + 63) / 64;
  dim3 grid(nb * (nb + 1) / 2, E);
  k_mirror_upper_bf16<<<grid, 256, 0, s>>>(static_cast<__nv_bfloat16*>(H), C);
  return cudaGetLastError();
}

}  // namespace gsq
