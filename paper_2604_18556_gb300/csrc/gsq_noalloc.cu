// Allocation-free entry point: the fused backward + Lion update of one step,
// for callers that cannot allocate device memory (a host application that owns
// a fixed memory pool, a plugin whose host forbids allocation, or code that
// runs while allocation is not allowed).  They pass the state and dL/dW^ in
// their own buffers; the kernel's only scratch -- the last-block counter and
// one double partial loss per thread block -- lives in the file-scope array
// below, which every GPU that loads this library holds until the process exits.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "gsq_internal.h"

namespace gsq {
namespace {

// 256 B of status words followed by one double per thread block.
constexpr size_t kNoAllocScratchBytes = 256 + 8 * 16384;      // 131,328 B
constexpr int64_t kNoAllocMaxBlocks = (kNoAllocScratchBytes - 256) / 8;
constexpr int64_t kNoAllocMaxWeights = kNoAllocMaxBlocks * kEwThreads * 4;  // 16,777,216
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

gsq_status na_fail(gsq_status st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  return set_last_error(st, buf);  // reported by gsq_last_error()
}

// Device address of g_noalloc_scratch, cached per device together with the ID of
// the CUDA context it was looked up in (the host-side name is only a stand-in,
// not a device address).  A context ID is never reused within a process, so
// after cudaDeviceReset, or when the caller makes another context current on
// the same device, the module is loaded anew and the ID no longer matches: the
// address is then looked up again instead of reusing a stale one.
typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long*);

struct ScratchSlot {
  unsigned long long ctx_id;
  unsigned char* addr;
};

std::mutex g_addr_mu;
ScratchSlot g_slot[kMaxDevices] = {};
CtxGetCurrentFn g_ctx_current = nullptr;
CtxGetIdFn g_ctx_id = nullptr;

gsq_status driver_fns() {
  if (g_ctx_current && g_ctx_id) return GSQ_OK;
  void* a = nullptr;
  void* b = nullptr;
  cudaDriverEntryPointQueryResult qa, qb;
  if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &a, 12000, cudaEnableDefault, &qa) !=
          cudaSuccess ||
      qa != cudaDriverEntryPointSuccess ||
      cudaGetDriverEntryPointByVersion("cuCtxGetId", &b, 12000, cudaEnableDefault, &qb) !=
          cudaSuccess ||
      qb != cudaDriverEntryPointSuccess)
    return na_fail(GSQ_ERR_CUDA, "driver entry points cuCtxGetCurrent / cuCtxGetId not found");
  g_ctx_current = reinterpret_cast<CtxGetCurrentFn>(a);
  g_ctx_id = reinterpret_cast<CtxGetIdFn>(b);
  return GSQ_OK;
}

gsq_status current_ctx_id(unsigned long long* id) {
  CUcontext ctx = nullptr;
  if (g_ctx_current(&ctx) != CUDA_SUCCESS || !ctx) return GSQ_ERR_CUDA;
  return g_ctx_id(ctx, id) == CUDA_SUCCESS ? GSQ_OK : GSQ_ERR_CUDA;
}

gsq_status scratch_address(int dev, unsigned char** out) {
  std::lock_guard<std::mutex> lk(g_addr_mu);
  gsq_status st = driver_fns();
  if (st != GSQ_OK) return st;
  unsigned long long id = 0;
  // No context is current before the first runtime call that needs one: the
  // lookup below makes the device's primary context current, then it has an ID.
  const bool have_ctx = current_ctx_id(&id) == GSQ_OK;
  if (have_ctx && g_slot[dev].addr && g_slot[dev].ctx_id == id) {
    *out = g_slot[dev].addr;
    return GSQ_OK;
  }
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
  if (e != cudaSuccess)
    return na_fail(GSQ_ERR_CUDA, "cudaGetSymbolAddress(scratch): %s", cudaGetErrorString(e));
  if (!have_ctx && current_ctx_id(&id) != GSQ_OK)
    return na_fail(GSQ_ERR_CUDA, "no current CUDA context after the scratch lookup");
  g_slot[dev].ctx_id = id;
  g_slot[dev].addr = static_cast<unsigned char*>(p);
  *out = g_slot[dev].addr;
  return GSQ_OK;
}

}  // namespace
}  // namespace gsq

using namespace gsq;

extern "C" GSQ_API gsq_status gsq_backward_update_noalloc(const gsq_backward_args* a, void* stream) {
  if (!a) return na_fail(GSQ_ERR_INVALID_ARG, "args is NULL");
  if (a->num_experts < 1 || a->out_features < 1 || a->in_features < 8 || a->in_features % 8)
    return na_fail(GSQ_ERR_SHAPE, "need E >= 1, R >= 1, C >= 8 with C %% 8 == 0");
  if (a->num_levels < 2 || a->num_levels > GSQ_MAX_LEVELS)
    return na_fail(GSQ_ERR_INVALID_ARG, "num_levels must be in [2, 8]");
  const int g = a->group_size;
  if (g < 4 || g > 128 || (g & (g - 1)) || a->in_features % g)
    return na_fail(GSQ_ERR_SHAPE, "group_size must be a power of two in [4, 128] dividing C");
  const int64_t n = static_cast<int64_t>(a->num_experts) * a->out_features * a->in_features;
  if (n > kNoAllocMaxWeights)
    return na_fail(GSQ_ERR_SHAPE,
                   "E*R*C = %lld exceeds the allocation-free limit of %lld weights "
                   "(%zu bytes of static scratch)",
                   static_cast<long long>(n), static_cast<long long>(kNoAllocMaxWeights),
                   kNoAllocScratchBytes);
  if (!a->W || !a->G || !a->logits || !a->m_logits || !a->scales || !a->m_scales)
    return na_fail(GSQ_ERR_INVALID_ARG, "W, G, logits, m_logits, scales and m_scales are required");
  if (a->w_dtype != GSQ_DTYPE_F32 && a->w_dtype != GSQ_DTYPE_BF16)
    return na_fail(GSQ_ERR_INVALID_ARG, "bad w_dtype");
  if (a->d_dtype != GSQ_DTYPE_F32 && a->d_dtype != GSQ_DTYPE_BF16)
    return na_fail(GSQ_ERR_INVALID_ARG, "bad d_dtype");
  if (a->flags & ~static_cast<uint32_t>(GSQ_FLAG_NO_NOISE))
    return na_fail(GSQ_ERR_INVALID_ARG, "flags: only GSQ_FLAG_NO_NOISE is accepted");
  if (a->step >= (1ull << 32)) return na_fail(GSQ_ERR_INVALID_ARG, "step must be < 2^32");
  if (!(a->tau > 0.f) || !std::isfinite(a->tau) || !std::isfinite(a->kappa))
    return na_fail(GSQ_ERR_INVALID_ARG, "need tau > 0 and finite kappa");
  for (int k = 1; k < a->num_levels; ++k)
    if (!(a->grid[k] > a->grid[k - 1])) return na_fail(GSQ_ERR_INVALID_ARG, "grid must ascend");

  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return na_fail(GSQ_ERR_CUDA, "cudaGetDevice: %s", cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices) return na_fail(GSQ_ERR_UNSUPPORTED, "device index %d", dev);
  unsigned char* scratch = nullptr;
  gsq_status st = scratch_address(dev, &scratch);
  if (st != GSQ_OK) return st;

  EwParams p;
  std::memset(&p, 0, sizeof(p));
  p.n = n;
  p.nq = n / 4;
  p.K = a->num_levels;
  p.nlev = a->num_levels;
  p.group = g;
  int lg = 0;
  while ((1 << lg) < g) ++lg;
  p.log2_group = lg;
  p.w_bf16 = a->w_dtype == GSQ_DTYPE_BF16;
  p.d_bf16 = a->d_dtype == GSQ_DTYPE_BF16;
  for (int k = 0; k < kMaxLevels; ++k) p.grid[k] = k < a->num_levels ? a->grid[k] : 0.f;
  p.logits = a->logits;
  p.m_logits = a->m_logits;
  p.scales = a->scales;
  p.m_scales = a->m_scales;
  p.W = a->W;
  p.G = a->G;
  const uint32_t key0 = static_cast<uint32_t>(a->seed), key1 = static_cast<uint32_t>(a->seed >> 32);
  for (uint32_t r = 0; r < 10; ++r) {
    p.keys.k0[r] = key0 + r * 0x9E3779B9u;
    p.keys.k1[r] = key1 + r * 0xBB67AE85u;
  }
  p.noise = (a->flags & GSQ_FLAG_NO_NOISE) ? 0 : 1;
  p.t = static_cast<uint32_t>(a->step);
  p.kappa_log2 = static_cast<float>(a->kappa * 1.4426950408889634);
  p.inv_tau = static_cast<float>(1.0 / a->tau);
  p.kappa_over_tau = static_cast<float>(static_cast<double>(a->kappa) / a->tau);
  p.lr_l = a->lr_logits;
  p.lr_s = a->lr_scales;
  p.b1 = a->beta1;
  p.b2 = a->beta2;
  p.wd_l = a->wd_logits;
  p.wd_s = a->wd_scales;
  p.lrwd_l = static_cast<float>(static_cast<double>(a->lr_logits) * a->wd_logits);
  p.lrwd_s = static_cast<float>(static_cast<double>(a->lr_scales) * a->wd_scales);
  p.scales_frozen = (a->lr_scales == 0.f && a->wd_scales == 0.f) ? 1 : 0;
  p.flags = reinterpret_cast<DevFlags*>(scratch);
  p.loss_partials = reinterpret_cast<double*>(scratch + 256);
  p.loss_out = a->loss_dev;

  // one quad per thread: one partial per block, at most kNoAllocMaxBlocks of them
  const int64_t blocks = (p.nq + kEwThreads - 1) / kEwThreads;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // the array keeps the previous call's contents: the counter must start at zero
  e = cudaMemsetAsync(scratch, 0, sizeof(DevFlags), s);
  if (e != cudaSuccess) return na_fail(GSQ_ERR_CUDA, "clear scratch: %s", cudaGetErrorString(e));
  e = launch_backward(p, static_cast<int>(blocks), s);
  if (e != cudaSuccess) return na_fail(GSQ_ERR_CUDA, "backward kernel: %s", cudaGetErrorString(e));
  return GSQ_OK;
}
