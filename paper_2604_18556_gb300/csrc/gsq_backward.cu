// The fused backward with direct global loads (k_backward): every variant
// (export, gradient accumulation) and every relaxation policy; the staged
// kernel for non-exporting steps is in gsq_staged.cu.
#include <cuda_bf16.h>

#include <type_traits>

#include "gsq_backward.cuh"
#include "gsq_internal.h"

namespace gsq {
namespace {

template <class Rx, bool kExport, bool kShift, bool kAcc>
__global__ void __launch_bounds__(kEwThreads, BwdOcc<Rx::L>::value) k_backward(const EwParams P) {
  constexpr int K = Rx::L;
  grid_dep_wait();
  grid_dep_launch();
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

template <class Rx, bool kShift>
void set_backward_carveout() {
  const auto attr = cudaFuncAttributePreferredSharedMemoryCarveout;
  cudaFuncSetAttribute(k_backward<Rx, false, kShift, false>, attr, 0);
  cudaFuncSetAttribute(k_backward<Rx, true, kShift, false>, attr, 0);
  cudaFuncSetAttribute(k_backward<Rx, false, kShift, true>, attr, 0);
  cudaFuncSetAttribute(k_backward<Rx, true, kShift, true>, attr, 0);
}

}  // namespace

int ew_backward_grid(int K, int num_sms, int mode) {
  int g = num_sms;
  with_relax(K, mode, [&](auto rx, auto sh) {
    using Rx = typename decltype(rx)::type;
    constexpr bool SH = decltype(sh)::value;
    set_backward_carveout<Rx, SH>();
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(
            &per_sm, reinterpret_cast<const void*>(k_backward<Rx, false, SH, false>), kEwThreads,
            0) != cudaSuccess ||
        per_sm < 1)
      per_sm = 1;
    g = per_sm * num_sms;
  });
  return g;
}

cudaError_t launch_backward(const EwParams& p, int grid, cudaStream_t s, bool pdl) {
  const bool export_mode = (p.grad_logits != nullptr) || (p.grad_scales != nullptr);
  const bool acc = p.acc_in_l != nullptr;
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
    if (export_mode)
      le = acc ? cudaLaunchKernelEx(&cfg, k_backward<Rx, true, SH, true>, p)
               : cudaLaunchKernelEx(&cfg, k_backward<Rx, true, SH, false>, p);
    else
      le = acc ? cudaLaunchKernelEx(&cfg, k_backward<Rx, false, SH, true>, p)
               : cudaLaunchKernelEx(&cfg, k_backward<Rx, false, SH, false>, p);
  });
  if (e != cudaSuccess) return e;
  return le != cudaSuccess ? le : cudaGetLastError();
}

}  // namespace gsq
