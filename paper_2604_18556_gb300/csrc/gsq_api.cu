// Host side of libgsq: the extern "C" entry points declared in include/gsq.h.
// Validates arguments, carves the caller's workspace, sequences the kernels on
// the caller's stream and keeps the per-layer bookkeeping (pending look-ahead
// forward, profiling events).  Never allocates device memory.
#include <cuda_runtime.h>
#include <nvtx3/nvToolsExt.h>

#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <new>
#include <string>
#include <unordered_map>
#include <unordered_set>
#include <vector>

#include "gsq_internal.h"

namespace gsq {
namespace {

constexpr uint64_t kMagic = 0x6773715f6c617972ull;  // "gsq_layr"
constexpr int kMaxPartials = 16384;
constexpr int kMaxProfileEvents = 8192;
constexpr int kGemmGroupN = 8;  // GEMM tile order: 8 output-tile columns per group
constexpr size_t kCanaryBytes = 256;
static_assert(GSQ_DIAG_SHIFT_BINS == kDiagShiftBins && GSQ_DIAG_MARGIN_BINS == kDiagMarginBins,
              "diagnostics bins");
constexpr double kLog2e = 1.4426950408889634;

thread_local std::string g_last_error;

gsq_status fail(gsq_status st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return st;
}

}  // namespace

gsq_status set_last_error(gsq_status st, const char* msg) {
  g_last_error = msg;
  return st;
}

namespace {

gsq_status cuda_fail(cudaError_t e, const char* what) {
  return fail(GSQ_ERR_CUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

// GSQ_FAULT_INJECT=<function>:<n>: the n-th call of <function> fails.
bool injected(const char* fn) {
  static std::once_flag once;
  static std::string target;
  static long nth = 0;
  static std::mutex mu;
  static std::unordered_map<std::string, long> calls;
  std::call_once(once, [] {
    const char* v = std::getenv("GSQ_FAULT_INJECT");
    if (!v) return;
    const char* colon = std::strchr(v, ':');
    if (!colon) return;
    target.assign(v, colon - v);
    nth = std::strtol(colon + 1, nullptr, 10);
  });
  if (target.empty() || target != fn) return false;
  std::lock_guard<std::mutex> lk(mu);
  return ++calls[target] == nth;
}

#define GSQ_INJECT(fn)                                                     \
  do {                                                                     \
    if (injected(fn)) return fail(GSQ_ERR_INJECTED, "%s: injected fault", fn); \
  } while (0)

size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

struct Layout {
  size_t flags, partials, logits, m_logits, scales, m_scales, W, H, D, G, kq_d, kq_sc, hscratch, j0;
  size_t D2;     // second D buffer (bf16 layers stepped with gsq_step): D of step t lives in
                 // buffer t mod 2, so a step can write the next D while its own is still read
  bool has_d2;
  size_t tok_b, tok_t, Y, acc_l, acc_s;  // per-step token batches (GSQ_CALIB_BATCHES)
  size_t code0, diag;                     // initial codes and diagnostics counters
  size_t total;
  // 256 canary bytes after every buffer (written at init, checked by gsq_sync_status)
  int ncanary;
  size_t canary[kMaxCanaries];
  const char* canary_of[kMaxCanaries];
};

struct Shape {
  int64_t E, R, C, n, ng;
  int K, group;
  int L;     // logits per weight: K, 5 with local shift, 2 with mask x sign
  int mode;  // GSQ_PARAM_*
  int64_t T;  // GSQ_CALIB_BATCHES: most tokens per micro-batch and expert
  bool kquant, d_bf16, w_bf16, x_mode, shift, mask_sign, batches;
  bool gram;  // GSQ_CALIB_BATCHES on the tensor cores: contract through H = X^T X
};

Shape shape_of(const gsq_layer_desc& d) {
  Shape s;
  s.E = d.num_experts;
  s.R = d.out_features;
  s.C = d.in_features;
  s.n = s.E * s.R * s.C;
  s.K = d.num_levels;
  s.group = d.group_size;
  s.ng = s.group > 0 ? s.n / s.group : 0;
  s.kquant = d.scale_mode == GSQ_SCALE_KQUANT2;
  s.d_bf16 = d.gemm_precision == GSQ_GEMM_BF16;
  s.w_bf16 = d.w_dtype == GSQ_DTYPE_BF16;
  s.x_mode = d.calib_kind == GSQ_CALIB_X;
  s.batches = d.calib_kind == GSQ_CALIB_BATCHES;
  s.T = s.batches ? d.n_tokens : 0;
  s.mode = d.param_mode;
  s.shift = d.param_mode == GSQ_PARAM_SHIFT5;
  s.mask_sign = d.param_mode == GSQ_PARAM_MASK_SIGN;
  s.L = s.shift ? 5 : (s.mask_sign ? 2 : s.K);
  // Per-step tokens on the tensor cores: G = 2 D X^T X either as Y = D X^T, G = 2 Y X
  // (4 R T C flops per expert) or through the micro-batch's Gram matrix, H = X^T X
  // from the tiles of its upper triangle (C^2 T; every tile with GSQ_TOKEN_SYM=0:
  // 2 C^2 T), then G = 2 D H (2 R C^2), whichever costs fewer flops at the
  // descriptor's token count (4096 x 4096 with 32,768 tokens: 0.69 against 2.2
  // TFLOP).  GSQ_TOKEN_ROUTE=direct|gram forces one.
  s.gram = false;
  if (s.batches && s.d_bf16) {
    const char* sv = std::getenv("GSQ_TOKEN_SYM");
    const bool sym = !(sv && std::atoi(sv) == 0);
    s.gram = sym ? s.C * (s.T + 2 * s.R) < 4 * s.R * s.T : s.C * (s.T + s.R) < 2 * s.R * s.T;
    if (const char* v = std::getenv("GSQ_TOKEN_ROUTE")) {
      if (std::strcmp(v, "direct") == 0) s.gram = false;
      if (std::strcmp(v, "gram") == 0) s.gram = true;
    }
  }
  return s;
}

Layout layout_of(const Shape& s) {
  Layout L;
  size_t off = 0;
  L.ncanary = 0;
  auto take = [&](size_t bytes, const char* name) {
    const size_t o = off;
    off += align256(bytes);
    L.canary_of[L.ncanary] = name;
    L.canary[L.ncanary++] = off;
    off += kCanaryBytes;
    return o;
  };
  const size_t n = static_cast<size_t>(s.n), ng = static_cast<size_t>(s.ng);
  L.flags = take(sizeof(DevFlags), "flags");
  L.partials = take(sizeof(double) * kMaxPartials, "partials");
  L.logits = take(4 * n * s.L, "logits");
  L.m_logits = take(4 * n * s.L, "m_logits");
  L.scales = take(4 * ng, "scales");
  L.m_scales = take(4 * ng, "m_scales");
  L.W = take(n * (s.w_bf16 ? 2 : 4), "W");
  // H: the layer's Gram matrices, or on the Gram route of per-step tokens the current
  // micro-batch's (bf16)
  L.H = !s.batches ? take(static_cast<size_t>(s.E) * s.C * s.C * (s.d_bf16 ? 2 : 4), "H")
                   : (s.gram ? take(static_cast<size_t>(s.E) * s.C * s.C * 2, "H") : off);
  L.D = take(n * (s.d_bf16 ? 2 : 4), "D");
  L.has_d2 = s.d_bf16 && !s.batches;
  L.D2 = L.has_d2 ? take(2 * n, "D2") : off;
  L.G = take(4 * n, "G");
  L.kq_d = s.kquant ? take(2 * (n / kSuperBlock), "kq_d") : off;
  L.kq_sc = s.kquant ? take(n / kSubBlock, "kq_sc") : off;
  L.hscratch = s.x_mode ? take(static_cast<size_t>(s.E) * s.C * s.C * 4, "hscratch") : off;
  L.j0 = s.shift ? take(n, "j0") : off;
  const size_t et = static_cast<size_t>(s.E) * static_cast<size_t>(s.T);
  L.tok_b = s.batches && s.d_bf16 && !s.gram ? take(2 * et * s.C, "tok_b") : off;
  L.tok_t = s.batches && s.d_bf16 ? take(2 * et * s.C, "tok_t") : off;
  L.Y = s.batches && !s.gram ? take((s.d_bf16 ? 2 : 4) * et * s.R, "Y") : off;
  L.acc_l = s.batches ? take(4 * n * s.L, "acc_l") : off;
  L.acc_s = s.batches ? take(4 * ng, "acc_s") : off;
  L.code0 = take(n, "code0");
  L.diag = take(8 * (kDiagShiftBins + kDiagMarginBins), "diag");
  L.total = off;
  return L;
}

CanaryList canary_list(const Layout& lay) {
  CanaryList c;
  c.count = lay.ncanary;
  for (int i = 0; i < lay.ncanary; ++i) c.off[i] = lay.canary[i];
  return c;
}

bool is_pow2(int v) { return v > 0 && (v & (v - 1)) == 0; }

gsq_status validate_desc(const gsq_layer_desc* d) {
  if (!d) return fail(GSQ_ERR_INVALID_ARG, "desc is NULL");
  if (d->num_experts < 1 || d->out_features < 1 || d->in_features < 8)
    return fail(GSQ_ERR_SHAPE, "need E >= 1, R >= 1, C >= 8 (got %d, %d, %d)", d->num_experts,
                d->out_features, d->in_features);
  if (d->in_features % 8 != 0) return fail(GSQ_ERR_SHAPE, "in_features %% 8 != 0 (%d)", d->in_features);
  const double n = static_cast<double>(d->num_experts) * d->out_features * d->in_features;
  if (n >= 1099511627776.0) return fail(GSQ_ERR_SHAPE, "E*R*C must be < 2^40");
  if (d->num_levels < 2 || d->num_levels > GSQ_MAX_LEVELS)
    return fail(GSQ_ERR_INVALID_ARG, "num_levels must be in [2, 8] (got %d)", d->num_levels);
  for (int k = 0; k < d->num_levels; ++k) {
    if (!std::isfinite(d->grid[k])) return fail(GSQ_ERR_INVALID_ARG, "grid[%d] is not finite", k);
    if (k > 0 && !(d->grid[k] > d->grid[k - 1]))
      return fail(GSQ_ERR_INVALID_ARG, "grid must be strictly ascending");
  }
  float qmax = 0.f;
  for (int k = 0; k < d->num_levels; ++k) qmax = std::fmax(qmax, std::fabs(d->grid[k]));
  if (!(qmax > 0.f)) return fail(GSQ_ERR_INVALID_ARG, "grid must have a nonzero level");
  if (!is_pow2(d->group_size) || d->group_size < 4 || d->group_size > 128)
    return fail(GSQ_ERR_SHAPE, "group_size must be a power of two in [4, 128] (got %d)", d->group_size);
  if (d->in_features % d->group_size != 0)
    return fail(GSQ_ERR_SHAPE, "in_features %% group_size != 0");
  if (d->w_dtype != GSQ_DTYPE_F32 && d->w_dtype != GSQ_DTYPE_BF16)
    return fail(GSQ_ERR_INVALID_ARG, "bad w_dtype %d", d->w_dtype);
  if (d->calib_kind != GSQ_CALIB_H && d->calib_kind != GSQ_CALIB_X &&
      d->calib_kind != GSQ_CALIB_BATCHES)
    return fail(GSQ_ERR_INVALID_ARG, "bad calib_kind %d", d->calib_kind);
  if (d->calib_kind == GSQ_CALIB_BATCHES &&
      (d->n_tokens < 8 || d->n_tokens > 2147483647LL || d->n_tokens % 8 != 0))
    return fail(GSQ_ERR_INVALID_ARG, "GSQ_CALIB_BATCHES needs n_tokens in [8, 2^31), a multiple of 8");
  if (d->calib_kind == GSQ_CALIB_X && (d->n_tokens < 1 || d->n_tokens > 2147483647LL))
    return fail(GSQ_ERR_INVALID_ARG, "n_tokens must be in [1, 2^31) for GSQ_CALIB_X");
  if (d->scale_mode != GSQ_SCALE_GROUP && d->scale_mode != GSQ_SCALE_KQUANT2)
    return fail(GSQ_ERR_INVALID_ARG, "bad scale_mode %d", d->scale_mode);
  if (d->scale_mode == GSQ_SCALE_KQUANT2) {
    if (d->group_size != kSubBlock) return fail(GSQ_ERR_SHAPE, "GSQ_SCALE_KQUANT2 needs group_size 16");
    if (d->in_features % kSuperBlock != 0)
      return fail(GSQ_ERR_SHAPE, "GSQ_SCALE_KQUANT2 needs in_features %% 256 == 0");
    if (d->lr_scales != 0.f || d->wd_scales != 0.f)
      return fail(GSQ_ERR_INVALID_ARG, "GSQ_SCALE_KQUANT2 scales are frozen: lr_scales = wd_scales = 0");
  }
  if (d->gemm_precision != GSQ_GEMM_BF16 && d->gemm_precision != GSQ_GEMM_F32)
    return fail(GSQ_ERR_INVALID_ARG, "bad gemm_precision %d", d->gemm_precision);
  if (d->flags & ~static_cast<uint32_t>(GSQ_FLAG_NO_NOISE | GSQ_FLAG_UNSTAGED))
    return fail(GSQ_ERR_INVALID_ARG, "unknown flags 0x%x", d->flags);
  if (d->param_mode != GSQ_PARAM_FULL && d->param_mode != GSQ_PARAM_SHIFT5 &&
      d->param_mode != GSQ_PARAM_MASK_SIGN)
    return fail(GSQ_ERR_INVALID_ARG, "bad param_mode %d", d->param_mode);
  if (d->param_mode == GSQ_PARAM_MASK_SIGN &&
      !(d->num_levels == 3 && d->grid[1] == 0.f && d->grid[0] == -d->grid[2]))
    return fail(GSQ_ERR_INVALID_ARG, "GSQ_PARAM_MASK_SIGN needs the grid {-a, 0, a}");
  const float hp[] = {d->init_bias, d->lr_logits, d->lr_scales, d->beta1, d->beta2, d->wd_logits, d->wd_scales};
  for (float v : hp)
    if (!std::isfinite(v)) return fail(GSQ_ERR_INVALID_ARG, "non-finite hyper-parameter");
  if (d->beta1 < 0.f || d->beta1 > 1.f || d->beta2 < 0.f || d->beta2 > 1.f)
    return fail(GSQ_ERR_INVALID_ARG, "betas must be in [0, 1]");
  if (d->lr_logits < 0.f || d->lr_scales < 0.f) return fail(GSQ_ERR_INVALID_ARG, "negative learning rate");
  if (d->index_offset % 8 != 0 || d->index_offset > (1ull << 62) - static_cast<uint64_t>(n))
    return fail(GSQ_ERR_INVALID_ARG, "index_offset must be a multiple of 8 below 2^62 - E*R*C");
  return GSQ_OK;
}

struct DeviceGuard {
  int prev = -1;
  bool switched = false;
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev) == cudaSuccess && prev != dev) switched = cudaSetDevice(dev) == cudaSuccess;
  }
  ~DeviceGuard() {
    if (switched) cudaSetDevice(prev);
  }
};

}  // namespace
}  // namespace gsq

using namespace gsq;

struct gsq_layer {
  uint64_t magic;
  gsq_layer_desc desc;
  Shape shape;
  Layout lay;
  uint8_t* ws;
  int device;
  int num_sms;
  int grid_fwd, grid_bwd;
  int grid_bwd_staged;  // TMA-staged backward (non-export steps); 0: not used
  int staged_plan;      // its staging plan
  bool tc;
  int tile_n;  // N of the tensor-core GEMM tile (128 or 256)
  int group_n; // column group of the GEMM's tile order
  int gemm_pair;      // 1: the loss GEMM runs on CTA pairs (cta_group::2)
  int test_stall;     // test hook (GSQ_TEST_STALL): 1 staged backward, 2 tensor-core GEMM
  bool pdl;           // step kernels launched as programmatic dependents of the one before
  bool token_sym;     // Gram route of per-step tokens: X^T X from its upper triangle
  bool g_valid; // the G buffer holds the last step's G
  size_t d_cur; // offset of the buffer holding the latest D written
  // pending forward (D valid for these arguments)
  bool d_ready;
  uint64_t d_step;
  float d_tau, d_kappa;
  // micro-batch sequence of gsq_step_tokens: the next call it accepts
  uint64_t mb_step;
  uint32_t mb_next, mb_count;
  // profiling
  bool profiling;
  std::vector<cudaEvent_t> ev;  // pairs
  std::vector<int> ev_kind;
  int ev_used;
  cudaStream_t last_stream;
};

namespace {

float* fptr(gsq_layer* L, size_t off) { return reinterpret_cast<float*>(L->ws + off); }

// Offset of the D buffer of noise counter t (forward pass t writes it, its loss
// contraction reads it).
size_t d_off(const gsq_layer* L, uint64_t t) {
  return (L->lay.has_d2 && (t & 1u)) ? L->lay.D2 : L->lay.D;
}

// Live handles, so a stale or twice-destroyed pointer is rejected without
// being dereferenced.
std::mutex g_live_mu;
std::unordered_set<const gsq_layer*> g_live;

bool valid(const gsq_layer* L) {
  if (!L) return false;
  std::lock_guard<std::mutex> lk(g_live_mu);
  return g_live.count(L) != 0 && L->magic == kMagic;
}

void register_live(const gsq_layer* L) {
  std::lock_guard<std::mutex> lk(g_live_mu);
  g_live.insert(L);
}

void unregister_live(const gsq_layer* L) {
  std::lock_guard<std::mutex> lk(g_live_mu);
  g_live.erase(L);
}

EwParams base_params(gsq_layer* L) {
  EwParams p;
  std::memset(&p, 0, sizeof(p));
  const Shape& s = L->shape;
  const gsq_layer_desc& d = L->desc;
  p.n = s.n;
  p.nq = s.n / 4;
  p.K = s.L;
  p.nlev = s.K;
  p.mode = s.mode;
  p.j0 = s.shift ? L->ws + L->lay.j0 : nullptr;
  p.group = s.group;
  int lg = 0;
  while ((1 << lg) < s.group) ++lg;
  p.log2_group = lg;
  p.w_bf16 = s.w_bf16;
  p.d_bf16 = s.d_bf16;
  for (int k = 0; k < kMaxLevels; ++k) p.grid[k] = k < s.K ? d.grid[k] : 0.f;
  p.logits = fptr(L, L->lay.logits);
  p.m_logits = fptr(L, L->lay.m_logits);
  p.scales = fptr(L, L->lay.scales);
  p.m_scales = fptr(L, L->lay.m_scales);
  p.W = L->ws + L->lay.W;
  p.D = L->ws + L->lay.D;
  p.G = fptr(L, L->lay.G);
  const uint32_t key0 = static_cast<uint32_t>(d.seed), key1 = static_cast<uint32_t>(d.seed >> 32);
  for (uint32_t r = 0; r < 10; ++r) {
    p.keys.k0[r] = key0 + r * 0x9E3779B9u;
    p.keys.k1[r] = key1 + r * 0xBB67AE85u;
  }
  p.noise = (d.flags & GSQ_FLAG_NO_NOISE) ? 0 : 1;
  p.index_base = d.index_offset;
  p.lr_l = d.lr_logits;
  p.lr_s = d.lr_scales;
  p.b1 = d.beta1;
  p.b2 = d.beta2;
  p.wd_l = d.wd_logits;
  p.wd_s = d.wd_scales;
  p.lrwd_l = static_cast<float>(static_cast<double>(d.lr_logits) * d.wd_logits);
  p.lrwd_s = static_cast<float>(static_cast<double>(d.lr_scales) * d.wd_scales);
  p.scales_frozen = (d.lr_scales == 0.f && d.wd_scales == 0.f) ? 1 : 0;
  p.loss_partials = reinterpret_cast<double*>(L->ws + L->lay.partials);
  p.flags = reinterpret_cast<DevFlags*>(L->ws + L->lay.flags);
  p.stall = L->test_stall == 1 ? 1 : 0;
  return p;
}

// Profiling events; in a stream being captured into a CUDA graph they become
// event-record nodes, so every replay of the graph re-times its kernels.
void prof_record(cudaEvent_t ev, cudaStream_t s) {
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(s, &cs) == cudaSuccess && cs == cudaStreamCaptureStatusActive)
    cudaEventRecordWithFlags(ev, s, cudaEventRecordExternal);
  else
    cudaEventRecord(ev, s);
}

// NVTX range names per kernel kind (visible in nsys / ncu timelines).
const char* const kKindName[GSQ_K_COUNT] = {"gsq:forward", "gsq:gemm",  "gsq:backward",
                                            "gsq:project", "gsq:pack",  "gsq:init",
                                            "gsq:tokens"};

void prof_begin(gsq_layer* L, int kind, cudaStream_t s, int& slot) {
  nvtxRangePushA(kKindName[kind]);
  slot = -1;
  if (!L->profiling || L->ev_used >= kMaxProfileEvents) return;
  const int i = L->ev_used;
  if (static_cast<int>(L->ev_kind.size()) <= i) {
    cudaEvent_t a, b;
    if (cudaEventCreate(&a) != cudaSuccess) return;
    if (cudaEventCreate(&b) != cudaSuccess) {
      cudaEventDestroy(a);
      return;
    }
    L->ev.push_back(a);
    L->ev.push_back(b);
    L->ev_kind.push_back(kind);
  }
  L->ev_kind[i] = kind;
  prof_record(L->ev[2 * i], s);
  slot = i;
  L->ev_used = i + 1;
}

void prof_end(gsq_layer* L, int slot, cudaStream_t s) {
  nvtxRangePop();
  if (slot < 0) return;
  prof_record(L->ev[2 * slot + 1], s);
  L->last_stream = s;
}

gsq_status launch_fwd(gsq_layer* L, uint64_t step, float tau, float kappa, float* what,
                      cudaStream_t s) {
  EwParams p = base_params(L);
  p.t = static_cast<uint32_t>(step);
  p.kappa_log2 = static_cast<float>(kappa * kLog2e);
  p.inv_tau = static_cast<float>(1.0 / tau);
  p.kappa_over_tau = static_cast<float>(static_cast<double>(kappa) / tau);
  p.what = what;
  p.D = L->ws + d_off(L, step);
  int slot;
  prof_begin(L, GSQ_K_FORWARD, s, slot);
  const cudaError_t e = launch_forward(p, L->grid_fwd, s);
  prof_end(L, slot, s);
  if (e != cudaSuccess) return cuda_fail(e, "forward kernel");
  L->d_cur = d_off(L, step);
  L->d_ready = true;
  L->d_step = step;
  L->d_tau = tau;
  L->d_kappa = kappa;
  return GSQ_OK;
}

gsq_status launch_gemm(gsq_layer* L, size_t doff, cudaStream_t s) {
  const Shape& sh = L->shape;
  int slot;
  prof_begin(L, GSQ_K_GEMM, s, slot);
  cudaError_t e;
  if (sh.d_bf16) {
    TcGemm g{};  // G = 2 D H (H symmetrised, so its rows are K-major columns)
    g.stall = L->test_stall == 2 ? 1 : 0;
    g.E = static_cast<int>(sh.E);
    g.M = static_cast<int>(sh.R);
    g.N = static_cast<int>(sh.C);
    g.K = static_cast<int>(sh.C);
    g.A = L->ws + doff;
    g.B = L->ws + L->lay.H;
    g.out = fptr(L, L->lay.G);
    g.out_bf16 = 0;
    g.alpha = 2.0f;
    g.flags = reinterpret_cast<DevFlags*>(L->ws + L->lay.flags);
    g.tile_n = L->tile_n;
    g.group_n = L->group_n;
    g.pair = L->gemm_pair;
    g.pdl = L->pdl ? 1 : 0;
    e = launch_tc_gemm(g, L->num_sms, s);
  } else {
    SimtGemm g;
    g.batch = static_cast<int>(sh.E);
    g.M = static_cast<int>(sh.R);
    g.N = static_cast<int>(sh.C);
    g.Kd = static_cast<int>(sh.C);
    g.A = L->ws + doff;
    g.sam = sh.C;
    g.sak = 1;
    g.sab = sh.R * sh.C;
    g.B = L->ws + L->lay.H;
    g.sbk = sh.C;
    g.sbn = 1;
    g.sbb = sh.C * sh.C;
    g.C = fptr(L, L->lay.G);
    g.ldc = sh.C;
    g.scb = sh.R * sh.C;
    g.alpha = 2.0f;
    g.bf16_inputs = 0;
    e = launch_simt_gemm(g, s);
  }
  prof_end(L, slot, s);
  if (e != cudaSuccess) return cuda_fail(e, "loss GEMM");
  return GSQ_OK;
}

size_t tensor_bytes(const gsq_layer* L, int which) {
  const Shape& s = L->shape;
  const size_t n = static_cast<size_t>(s.n), ng = static_cast<size_t>(s.ng);
  switch (which) {
    case GSQ_T_LOGITS:
    case GSQ_T_MOM_LOGITS: return 4 * n * s.L;
    case GSQ_T_SCALES:
    case GSQ_T_MOM_SCALES: return 4 * ng;
    case GSQ_T_D: return n * (s.d_bf16 ? 2 : 4);
    case GSQ_T_G: return 4 * n;
    case GSQ_T_W: return n * (s.w_bf16 ? 2 : 4);
    case GSQ_T_H: return s.batches && !s.gram ? 0
                                              : static_cast<size_t>(s.E) * s.C * s.C * (s.d_bf16 ? 2 : 4);
    case GSQ_T_KQ_D: return s.kquant ? 2 * (n / kSuperBlock) : 0;
    case GSQ_T_KQ_SC: return s.kquant ? n / kSubBlock : 0;
    case GSQ_T_J0: return s.shift ? n : 0;
    default: return 0;
  }
}

size_t tensor_offset(const gsq_layer* L, int which) {
  switch (which) {
    case GSQ_T_LOGITS: return L->lay.logits;
    case GSQ_T_MOM_LOGITS: return L->lay.m_logits;
    case GSQ_T_SCALES: return L->lay.scales;
    case GSQ_T_MOM_SCALES: return L->lay.m_scales;
    case GSQ_T_D: return L->d_cur;
    case GSQ_T_G: return L->lay.G;
    case GSQ_T_W: return L->lay.W;
    case GSQ_T_H: return L->lay.H;
    case GSQ_T_KQ_D: return L->lay.kq_d;
    case GSQ_T_KQ_SC: return L->lay.kq_sc;
    case GSQ_T_J0: return L->lay.j0;
    default: return 0;
  }
}

size_t code_section_bytes(int64_t n, int K) {
  const int bits = K <= 4 ? 2 : 3;
  const size_t raw = static_cast<size_t>((n + 31) / 32) * 4 * bits;
  return (raw + 15) / 16 * 16;
}

size_t packed_bytes(const gsq_layer* L) {
  const Shape& s = L->shape;
  if (s.kquant) return static_cast<size_t>(s.n / kSuperBlock) * kKqRecord;
  return code_section_bytes(s.n, s.K) + 2 * static_cast<size_t>(s.ng);
}

}  // namespace

extern "C" {

gsq_status gsq_workspace_size(const gsq_layer_desc* desc, size_t* bytes) {
  GSQ_INJECT("gsq_workspace_size");
  if (!bytes) return fail(GSQ_ERR_INVALID_ARG, "bytes is NULL");
  const gsq_status st = validate_desc(desc);
  if (st != GSQ_OK) return st;
  *bytes = layout_of(shape_of(*desc)).total;
  return GSQ_OK;
}

gsq_status gsq_init_layer(const gsq_layer_desc* desc, void* workspace, size_t bytes, void* stream,
                          gsq_layer** out) {
  GSQ_INJECT("gsq_init_layer");
  if (!out) return fail(GSQ_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  gsq_status st = validate_desc(desc);
  if (st != GSQ_OK) return st;
  if (!desc->W || (!desc->calib && desc->calib_kind != GSQ_CALIB_BATCHES))
    return fail(GSQ_ERR_INVALID_ARG, "W and calib must be device pointers");
  if (!workspace) return fail(GSQ_ERR_WORKSPACE, "workspace is NULL");
  if (reinterpret_cast<uintptr_t>(workspace) % 256 != 0)
    return fail(GSQ_ERR_WORKSPACE, "workspace must be 256-byte aligned");
  const Shape sh = shape_of(*desc);
  const Layout lay = layout_of(sh);
  if (bytes < lay.total)
    return fail(GSQ_ERR_WORKSPACE, "workspace too small: %zu < %zu bytes", bytes, lay.total);

  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  cudaDeviceProp prop;
  e = cudaGetDeviceProperties(&prop, dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDeviceProperties");
  if (prop.major != 10 || prop.minor != 3)
    return fail(GSQ_ERR_UNSUPPORTED, "libgsq is built for sm_103 (found sm_%d%d)", prop.major, prop.minor);
  const bool tc = tc_gemm_supported(dev);
  if (sh.d_bf16 && !tc) return fail(GSQ_ERR_UNSUPPORTED, "tensor-map encoder unavailable for the bf16 GEMM");

  gsq_layer* L = new (std::nothrow) gsq_layer();
  if (!L) return fail(GSQ_ERR_INVALID_ARG, "host allocation failed");
  L->magic = kMagic;
  L->desc = *desc;
  L->desc.W = nullptr;      // borrowed pointers are not kept
  L->desc.calib = nullptr;
  L->shape = sh;
  L->lay = lay;
  L->ws = static_cast<uint8_t*>(workspace);
  L->device = dev;
  L->num_sms = prop.multiProcessorCount;
  L->tc = tc;
  L->g_valid = false;
  L->d_cur = lay.D;
  L->d_ready = false;
  L->mb_step = 0;
  L->mb_next = 0;
  L->mb_count = 0;
  L->profiling = false;
  L->ev_used = 0;
  L->last_stream = nullptr;
  const int64_t nq_blocks = (sh.n / 4 + kEwThreads - 1) / kEwThreads;
  auto clamp_grid = [&](int g) {
    int64_t v = g < nq_blocks ? g : nq_blocks;
    if (v > kMaxPartials) v = kMaxPartials;
    return static_cast<int>(v < 1 ? 1 : v);
  };
  L->grid_fwd = clamp_grid(ew_grid_size(sh.L, 0, L->num_sms, sh.mode));
  L->grid_bwd = clamp_grid(ew_grid_size(sh.L, 1, L->num_sms, sh.mode));
  {
    int lg = 0;
    while ((1 << lg) < sh.group) ++lg;
    const int frozen = (desc->lr_scales == 0.f && desc->wd_scales == 0.f) ? 1 : 0;
    L->staged_plan = 0;
    L->grid_bwd_staged =
        (desc->flags & GSQ_FLAG_UNSTAGED)
            ? 0
            : ew_staged_grid(sh.L, sh.mode, sh.w_bf16, lg, frozen, L->num_sms, &L->staged_plan);
    // staging pays only where every block gets more than one tile to overlap
    // (a plan forced through GSQ_STAGED_PLAN applies at any size)
    const bool forced = std::getenv("GSQ_STAGED_PLAN") != nullptr;
    if (L->grid_bwd_staged > 0 && !forced && nq_blocks <= L->grid_bwd_staged)
      L->grid_bwd_staged = 0;
    if (L->grid_bwd_staged > 0) L->grid_bwd_staged = clamp_grid(L->grid_bwd_staged);
  }
  // CTA pairs by default (at the same tile width measured 1-4% faster than single CTAs on the 4096 x 4096,
  // 4096 x 14336 and 64-expert layers); GSQ_GEMM_PAIR=0 selects single CTAs
  // (1: pairs or clusters of two pairs by the wave rule of tc_gemm_cluster_mode);
  // GSQ_GEMM_PAIR=1 forces plain pairs, =2 clusters of two pairs
  L->gemm_pair = 1;
  if (const char* gp = std::getenv("GSQ_GEMM_PAIR")) {
    const int v = std::atoi(gp);
    L->gemm_pair = v == 0 ? 0 : (v == 2 ? 2 : 3);
  }
  // Test hook for the bounded device-side waits: GSQ_TEST_STALL=backward makes the staged
  // backward skip one stage fill, =gemm makes the tensor-core GEMM skip its first k-block;
  // the waits on it give up after 2 s and gsq_sync_status reports GSQ_ERR_TIMEOUT.
  L->test_stall = 0;
  if (const char* ts = std::getenv("GSQ_TEST_STALL"))
    L->test_stall = std::strcmp(ts, "backward") == 0 ? 1 : (std::strcmp(ts, "gemm") == 0 ? 2 : 0);
  L->tile_n = tc_gemm_tile_n(static_cast<int>(sh.E), static_cast<int>(sh.R), static_cast<int>(sh.C),
                             L->num_sms, L->gemm_pair);
  if (const char* tn = std::getenv("GSQ_GEMM_TILE_N")) {   // 128, 224 or 256: override the choice
    const int v = std::atoi(tn);
    if (v == 128 || v == 224 || v == 256) L->tile_n = v;
  }
  // The step's tensor-core GEMMs and backward kernels are launched as programmatic
  // dependents: each is scheduled while the kernel before it drains and waits for it
  // (griddepcontrol) before touching memory. GSQ_PDL=0 launches them plainly.
  L->pdl = true;
  if (const char* pv = std::getenv("GSQ_PDL")) L->pdl = std::atoi(pv) != 0;
  // The Gram route forms X^T X from the tiles of its upper triangle and mirrors them
  // (half the flops); GSQ_TOKEN_SYM=0 computes every tile.
  L->token_sym = true;
  if (const char* sv = std::getenv("GSQ_TOKEN_SYM")) L->token_sym = std::atoi(sv) != 0;
  L->group_n = kGemmGroupN;
  if (const char* gn = std::getenv("GSQ_GEMM_GROUP_N")) {  // tile-order column group (0: none)
    const int v = std::atoi(gn);
    if (v >= 0 && v <= 1024) L->group_n = v;
  }
  // An H-based layer's loss contraction has one shape: settle pairs or clusters of pairs
  // once here rather than on every launch (token layers decide per contraction).
  if (L->gemm_pair == 1 && sh.d_bf16 && !sh.batches)
    L->gemm_pair = tc_gemm_cluster_mode(static_cast<int>(sh.E), static_cast<int>(sh.R),
                                        static_cast<int>(sh.C), L->tile_n, L->num_sms);

  cudaStream_t s = static_cast<cudaStream_t>(stream);
  DevFlags* flags = reinterpret_cast<DevFlags*>(L->ws + lay.flags);
  auto bail = [&](gsq_status code) {
    delete L;
    return code;
  };
  if ((e = cudaMemsetAsync(flags, 0, sizeof(DevFlags), s)) != cudaSuccess)
    return bail(cuda_fail(e, "clear flags"));
  if ((e = launch_canaries(L->ws, canary_list(lay), 1, flags, s)) != cudaSuccess)
    return bail(cuda_fail(e, "write canaries"));
  const size_t wbytes = static_cast<size_t>(sh.n) * (sh.w_bf16 ? 2 : 4);
  if ((e = cudaMemcpyAsync(L->ws + lay.W, desc->W, wbytes, cudaMemcpyDeviceToDevice, s)) != cudaSuccess)
    return bail(cuda_fail(e, "copy W"));
  if ((e = launch_nonfinite_scan(L->ws + lay.W, sh.n, sh.w_bf16, &flags->nonfinite, s)) != cudaSuccess)
    return bail(cuda_fail(e, "scan W"));
  if (!sh.batches) {
    const int64_t calib_count = sh.x_mode ? sh.E * desc->n_tokens * sh.C : sh.E * sh.C * sh.C;
    if ((e = launch_nonfinite_scan(desc->calib, calib_count, 0, &flags->nonfinite, s)) != cudaSuccess)
      return bail(cuda_fail(e, "scan calib"));
  }

  int slot;
  prof_begin(L, GSQ_K_INIT, s, slot);
  const float* hsrc = desc->calib;
  if (sh.x_mode) {
    SimtGemm g;  // H[e] = X[e]^T X[e]
    g.batch = static_cast<int>(sh.E);
    g.M = static_cast<int>(sh.C);
    g.N = static_cast<int>(sh.C);
    g.Kd = static_cast<int>(desc->n_tokens);
    g.A = desc->calib;
    g.sam = 1;
    g.sak = sh.C;
    g.sab = desc->n_tokens * sh.C;
    g.B = desc->calib;
    g.sbk = sh.C;
    g.sbn = 1;
    g.sbb = desc->n_tokens * sh.C;
    g.C = fptr(L, lay.hscratch);
    g.ldc = sh.C;
    g.scb = sh.C * sh.C;
    g.alpha = 1.0f;
    g.bf16_inputs = 0;
    if ((e = launch_simt_gemm(g, s)) != cudaSuccess) return bail(cuda_fail(e, "X^T X"));
    hsrc = fptr(L, lay.hscratch);
  }
  if (!sh.batches &&
      (e = launch_symmetrize(hsrc, L->ws + lay.H, static_cast<int>(sh.E), static_cast<int>(sh.C),
                             sh.d_bf16, s)) != cudaSuccess)
    return bail(cuda_fail(e, "symmetrise H"));

  InitParams ip;
  std::memset(&ip, 0, sizeof(ip));
  ip.n = sh.n;
  ip.K = sh.K;
  ip.group = sh.group;
  ip.kquant = sh.kquant;
  ip.w_bf16 = sh.w_bf16;
  for (int k = 0; k < kMaxLevels; ++k) ip.grid[k] = k < sh.K ? desc->grid[k] : 0.f;
  ip.init_bias = desc->init_bias;
  ip.W = L->ws + lay.W;
  ip.logits = fptr(L, lay.logits);
  ip.m_logits = fptr(L, lay.m_logits);
  ip.scales = fptr(L, lay.scales);
  ip.m_scales = fptr(L, lay.m_scales);
  ip.kq_d = sh.kquant ? reinterpret_cast<uint16_t*>(L->ws + lay.kq_d) : nullptr;
  ip.kq_sc = sh.kquant ? reinterpret_cast<int8_t*>(L->ws + lay.kq_sc) : nullptr;
  ip.j0 = sh.shift ? L->ws + lay.j0 : nullptr;
  ip.code0 = L->ws + lay.code0;
  ip.mask_sign = sh.mask_sign;
  if ((e = launch_init_state(ip, L->num_sms, s)) != cudaSuccess) return bail(cuda_fail(e, "init state"));
  prof_end(L, slot, s);

  unsigned int bad = 0;
  if ((e = cudaMemcpyAsync(&bad, &flags->nonfinite, sizeof(bad), cudaMemcpyDeviceToHost, s)) != cudaSuccess)
    return bail(cuda_fail(e, "read scan result"));
  if ((e = cudaStreamSynchronize(s)) != cudaSuccess) return bail(cuda_fail(e, "init"));
  if (bad) return bail(fail(GSQ_ERR_NONFINITE, "W or calib holds %u non-finite values", bad));
  register_live(L);
  *out = L;
  return GSQ_OK;
}

gsq_status gsq_step(gsq_layer* L, uint64_t step, float tau, float kappa, float next_tau,
                    float next_kappa, void* stream, float* loss_dev, float* grad_logits_dev,
                    float* grad_scales_dev) {
  GSQ_INJECT("gsq_step");
  if (!valid(L)) return fail(GSQ_ERR_INVALID_ARG, "invalid layer handle");
  if (L->shape.batches)
    return fail(GSQ_ERR_INVALID_ARG, "GSQ_CALIB_BATCHES layers step with gsq_step_tokens");
  if (step >= (1ull << 32)) return fail(GSQ_ERR_INVALID_ARG, "step must be < 2^32");
  if (!(tau > 0.f) || !std::isfinite(tau) || !std::isfinite(kappa))
    return fail(GSQ_ERR_INVALID_ARG, "need tau > 0 and finite kappa");
  const bool export_mode = grad_logits_dev || grad_scales_dev;
  const bool lookahead = !export_mode && next_tau > 0.f;
  if (lookahead) {
    if (!std::isfinite(next_tau) || !std::isfinite(next_kappa))
      return fail(GSQ_ERR_INVALID_ARG, "next_tau / next_kappa must be finite");
    if (step + 1 >= (1ull << 32)) return fail(GSQ_ERR_INVALID_ARG, "step + 1 must be < 2^32");
  }
  DeviceGuard guard(L->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  gsq_status st;
  if (!(L->d_ready && L->d_step == step && L->d_tau == tau && L->d_kappa == kappa)) {
    if ((st = launch_fwd(L, step, tau, kappa, nullptr, s)) != GSQ_OK) return st;
  }
  if ((st = launch_gemm(L, d_off(L, step), s)) != GSQ_OK) return st;

  EwParams p = base_params(L);
  p.t = static_cast<uint32_t>(step);
  p.kappa_log2 = static_cast<float>(kappa * kLog2e);
  p.inv_tau = static_cast<float>(1.0 / tau);
  p.kappa_over_tau = static_cast<float>(static_cast<double>(kappa) / tau);
  p.lookahead = lookahead ? 1 : 0;
  if (lookahead) {
    p.t_next = static_cast<uint32_t>(step + 1);
    p.kappa_log2_next = static_cast<float>(next_kappa * kLog2e);
    p.inv_tau_next = static_cast<float>(1.0 / next_tau);
  }
  p.D = L->ws + d_off(L, step + 1);  // the look-ahead's D
  p.grad_logits = grad_logits_dev;
  p.grad_scales = grad_scales_dev;
  p.loss_out = loss_dev;
  int slot;
  cudaError_t e;
  prof_begin(L, GSQ_K_BACKWARD, s, slot);
  e = (!export_mode && L->grid_bwd_staged > 0)
          ? launch_backward_staged(p, L->grid_bwd_staged, L->staged_plan, s, L->pdl)
          : launch_backward(p, L->grid_bwd, s, L->pdl);
  prof_end(L, slot, s);
  if (e != cudaSuccess) return cuda_fail(e, "backward kernel");
  L->g_valid = true;
  if (lookahead) {
    L->d_cur = d_off(L, step + 1);
    L->d_ready = true;
    L->d_step = step + 1;
    L->d_tau = next_tau;
    L->d_kappa = next_kappa;
  } else if (!export_mode) {
    L->d_ready = false;
  }
  return GSQ_OK;
}

gsq_status gsq_step_tokens(gsq_layer* L, uint64_t step, uint32_t micro, uint32_t n_micro,
                           float tau, float kappa, float next_tau, float next_kappa,
                           const float* X_dev, int64_t n_tokens, void* stream, float* loss_dev) {
  GSQ_INJECT("gsq_step_tokens");
  if (!valid(L)) return fail(GSQ_ERR_INVALID_ARG, "invalid layer handle");
  const Shape& sh = L->shape;
  if (!sh.batches) return fail(GSQ_ERR_INVALID_ARG, "gsq_step_tokens needs a GSQ_CALIB_BATCHES layer");
  if (!X_dev) return fail(GSQ_ERR_INVALID_ARG, "X_dev is NULL");
  if (n_tokens < 8 || n_tokens > sh.T || n_tokens % 8 != 0)
    return fail(GSQ_ERR_INVALID_ARG, "n_tokens must be a multiple of 8 in [8, %lld]",
                static_cast<long long>(sh.T));
  if (n_micro < 1 || micro >= n_micro) return fail(GSQ_ERR_INVALID_ARG, "need micro < n_micro");
  const uint64_t t = step * n_micro + micro;  // noise counter of this forward pass
  if (step >= (1ull << 32) || t + 1 >= (1ull << 32))
    return fail(GSQ_ERR_INVALID_ARG, "step * n_micro + micro + 1 must be < 2^32");
  if (!(tau > 0.f) || !std::isfinite(tau) || !std::isfinite(kappa))
    return fail(GSQ_ERR_INVALID_ARG, "need tau > 0 and finite kappa");
  const bool last = micro + 1 == n_micro;
  const bool lookahead = !last || next_tau > 0.f;
  if (last && lookahead && (!std::isfinite(next_tau) || !std::isfinite(next_kappa)))
    return fail(GSQ_ERR_INVALID_ARG, "next_tau / next_kappa must be finite");
  if (micro > 0 && !(L->mb_step == step && L->mb_next == micro && L->mb_count == n_micro))
    return fail(GSQ_ERR_STATE, "micro-batches of a step must be issued in order from 0");
  DeviceGuard guard(L->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  gsq_status st;
  if (!(L->d_ready && L->d_step == t && L->d_tau == tau && L->d_kappa == kappa)) {
    if ((st = launch_fwd(L, t, tau, kappa, nullptr, s)) != GSQ_OK) return st;
  }

  // loss contraction on this micro-batch's tokens: Y = D X^T, G = 2 Y X, or on the Gram
  // route H = X^T X, G = 2 D H (the same G = 2 D X^T X in fewer flops when T > C)
  const int E = static_cast<int>(sh.E), R = static_cast<int>(sh.R), C = static_cast<int>(sh.C);
  const int T = static_cast<int>(n_tokens);
  int slot;
  cudaError_t e = cudaSuccess;
  void* Xb = L->ws + L->lay.tok_b;
  void* Xt = L->ws + L->lay.tok_t;
  if (sh.d_bf16) {
    prof_begin(L, GSQ_K_TOKENS, s, slot);
    e = launch_tokens_bf16(X_dev, sh.gram ? nullptr : Xb, Xt, E, T, C, T, s);
    prof_end(L, slot, s);
    if (e != cudaSuccess) return cuda_fail(e, "token conversion");
  }
  prof_begin(L, GSQ_K_GEMM, s, slot);
  if (sh.d_bf16) {
    TcGemm g{};
    g.stall = L->test_stall == 2 ? 1 : 0;
    g.flags = reinterpret_cast<DevFlags*>(L->ws + L->lay.flags);
    g.tile_n = 0;
    g.group_n = L->group_n;
    g.pair = L->gemm_pair;
    g.pdl = L->pdl ? 1 : 0;
    g.E = E;
    if (sh.gram) {
      void* Hj = L->ws + L->lay.H;
      if (e == cudaSuccess) {  // H[e] = X[e]^T X[e]  (M = N = C, K = T), bf16 out: the
        g.M = C; g.N = C; g.K = T;  // tiles of the upper triangle, then its mirror below
        g.A = Xt;
        g.B = Xt;
        g.out = Hj;
        g.out_bf16 = 1;
        g.alpha = 1.0f;
        g.sym = L->token_sym ? 1 : 0;
        e = launch_tc_gemm(g, L->num_sms, s);
        if (e == cudaSuccess && g.sym) e = launch_mirror_upper_bf16(Hj, E, C, s);
        g.sym = 0;
      }
      if (e == cudaSuccess) {  // G[e] = 2 D[e] H[e]  (N = C, K = C; H symmetric), fp32 out
        g.M = R; g.N = C; g.K = C;
        g.A = L->ws + L->lay.D;
        g.B = Hj;
        g.out = fptr(L, L->lay.G);
        g.out_bf16 = 0;
        g.alpha = 2.0f;
        e = launch_tc_gemm(g, L->num_sms, s);
      }
    }
    if (!sh.gram && e == cudaSuccess) {  // Y[e] = D[e] X[e]^T  (N = T, K = C), bf16 out
      g.M = R; g.N = T; g.K = C;
      g.A = L->ws + L->lay.D;
      g.B = Xb;
      g.out = L->ws + L->lay.Y;
      g.out_bf16 = 1;
      g.alpha = 1.0f;
      e = launch_tc_gemm(g, L->num_sms, s);
    }
    if (!sh.gram && e == cudaSuccess) {  // G[e] = 2 Y[e] X[e]  (N = C, K = T), fp32 out
      g.M = R; g.N = C; g.K = T;
      g.A = L->ws + L->lay.Y;
      g.B = Xt;
      g.out = fptr(L, L->lay.G);
      g.out_bf16 = 0;
      g.alpha = 2.0f;
      e = launch_tc_gemm(g, L->num_sms, s);
    }
  } else {
    SimtGemm g;  // Y[e][r][t] = sum_c D[e][r][c] X[e][t][c]
    g.batch = E;
    g.M = R; g.N = T; g.Kd = C;
    g.A = L->ws + L->lay.D; g.sam = C; g.sak = 1; g.sab = static_cast<int64_t>(R) * C;
    g.B = X_dev; g.sbk = 1; g.sbn = C; g.sbb = static_cast<int64_t>(T) * C;
    g.C = fptr(L, L->lay.Y); g.ldc = T; g.scb = static_cast<int64_t>(R) * T;
    g.alpha = 1.0f;
    g.bf16_inputs = 0;
    e = launch_simt_gemm(g, s);
    if (e == cudaSuccess) {  // G[e][r][c] = 2 sum_t Y[e][r][t] X[e][t][c]
      g.M = R; g.N = C; g.Kd = T;
      g.A = fptr(L, L->lay.Y); g.sam = T; g.sak = 1; g.sab = static_cast<int64_t>(R) * T;
      g.B = X_dev; g.sbk = C; g.sbn = 1; g.sbb = static_cast<int64_t>(T) * C;
      g.C = fptr(L, L->lay.G); g.ldc = C; g.scb = static_cast<int64_t>(R) * C;
      g.alpha = 2.0f;
      e = launch_simt_gemm(g, s);
    }
  }
  prof_end(L, slot, s);
  if (e != cudaSuccess) return cuda_fail(e, "token loss GEMMs");

  EwParams p = base_params(L);
  p.t = static_cast<uint32_t>(t);
  p.kappa_log2 = static_cast<float>(kappa * kLog2e);
  p.inv_tau = static_cast<float>(1.0 / tau);
  p.kappa_over_tau = static_cast<float>(static_cast<double>(kappa) / tau);
  const float nt = last ? next_tau : tau, nk = last ? next_kappa : kappa;
  p.lookahead = lookahead ? 1 : 0;
  if (lookahead) {
    p.t_next = static_cast<uint32_t>(t + 1);
    p.kappa_log2_next = static_cast<float>(nk * kLog2e);
    p.inv_tau_next = static_cast<float>(1.0 / nt);
  }
  float* acc_l = fptr(L, L->lay.acc_l);
  float* acc_s = fptr(L, L->lay.acc_s);
  if (!last) {  // export this micro-batch's gradient into the accumulator
    p.grad_logits = acc_l;
    p.grad_scales = acc_s;
  }
  if (micro > 0) {  // add the earlier micro-batches' sum; the last one takes the mean
    p.acc_in_l = acc_l;
    p.acc_in_s = p.scales_frozen ? nullptr : acc_s;
    p.acc_scale = last ? static_cast<float>(1.0 / n_micro) : 1.0f;
  }
  p.loss_out = loss_dev;
  prof_begin(L, GSQ_K_BACKWARD, s, slot);
  e = launch_backward(p, L->grid_bwd, s, L->pdl);
  prof_end(L, slot, s);
  if (e != cudaSuccess) return cuda_fail(e, "backward kernel");
  L->g_valid = true;
  if (lookahead) {
    L->d_ready = true;
    L->d_step = t + 1;
    L->d_tau = nt;
    L->d_kappa = nk;
  } else {
    L->d_ready = false;
  }
  L->mb_step = step;
  L->mb_next = last ? 0 : micro + 1;
  L->mb_count = n_micro;
  return GSQ_OK;
}

gsq_status gsq_forward(gsq_layer* L, uint64_t step, float tau, float kappa, void* stream,
                       float* what_dev) {
  GSQ_INJECT("gsq_forward");
  if (!valid(L)) return fail(GSQ_ERR_INVALID_ARG, "invalid layer handle");
  if (step >= (1ull << 32)) return fail(GSQ_ERR_INVALID_ARG, "step must be < 2^32");
  if (!(tau > 0.f) || !std::isfinite(tau) || !std::isfinite(kappa))
    return fail(GSQ_ERR_INVALID_ARG, "need tau > 0 and finite kappa");
  DeviceGuard guard(L->device);
  return launch_fwd(L, step, tau, kappa, what_dev, static_cast<cudaStream_t>(stream));
}

gsq_status gsq_init_logits(gsq_layer* L, const uint8_t* codes_dev, const float* eps_dev, float alpha,
                           float sigma, void* stream) {
  GSQ_INJECT("gsq_init_logits");
  if (!valid(L)) return fail(GSQ_ERR_INVALID_ARG, "invalid layer handle");
  if (!codes_dev) return fail(GSQ_ERR_INVALID_ARG, "codes_dev is NULL");
  if (!std::isfinite(alpha) || !std::isfinite(sigma))
    return fail(GSQ_ERR_INVALID_ARG, "alpha and sigma must be finite");
  DeviceGuard guard(L->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const Shape& sh = L->shape;
  InitCodesParams p;
  std::memset(&p, 0, sizeof(p));
  p.n = sh.n;
  p.K = sh.K;
  p.mode = sh.mode;
  for (int k = 0; k < kMaxLevels; ++k) p.grid[k] = k < sh.K ? L->desc.grid[k] : 0.f;
  p.codes = codes_dev;
  p.eps = eps_dev;
  p.alpha = alpha;
  p.sigma = sigma;
  p.logits = fptr(L, L->lay.logits);
  p.m_logits = fptr(L, L->lay.m_logits);
  p.j0 = sh.shift ? L->ws + L->lay.j0 : nullptr;
  p.code0 = L->ws + L->lay.code0;
  int slot;
  prof_begin(L, GSQ_K_INIT, s, slot);
  const cudaError_t e = launch_init_from_codes(p, L->num_sms, s);
  prof_end(L, slot, s);
  if (e != cudaSuccess) return cuda_fail(e, "init from codes");
  L->d_ready = false;
  return GSQ_OK;
}

gsq_status gsq_diagnose(gsq_layer* L, float tau, float kappa, void* stream, gsq_diagnostics* out) {
  GSQ_INJECT("gsq_diagnose");
  if (!valid(L)) return fail(GSQ_ERR_INVALID_ARG, "invalid layer handle");
  if (!out) return fail(GSQ_ERR_INVALID_ARG, "out is NULL");
  if (!(tau > 0.f) || !std::isfinite(tau) || !std::isfinite(kappa))
    return fail(GSQ_ERR_INVALID_ARG, "need tau > 0 and finite kappa");
  DeviceGuard guard(L->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const Shape& sh = L->shape;
  DiagParams p;
  p.n = sh.n;
  p.K = sh.L;
  p.nlev = sh.K;
  p.mask_sign = sh.mask_sign;
  p.j0 = sh.shift ? L->ws + L->lay.j0 : nullptr;
  p.logits = fptr(L, L->lay.logits);
  p.code0 = L->ws + L->lay.code0;
  p.kappa_over_tau = static_cast<double>(kappa) / tau;
  p.hist = reinterpret_cast<unsigned long long*>(L->ws + L->lay.diag);
  p.partials = reinterpret_cast<double*>(L->ws + L->lay.partials);
  const int grid = L->grid_fwd;
  unsigned long long hist[kDiagShiftBins + kDiagMarginBins];
  std::vector<double> parts(static_cast<size_t>(grid));
  cudaError_t e = cudaMemsetAsync(p.hist, 0, sizeof(hist), s);
  if (e == cudaSuccess) e = launch_diagnose(p, grid, s);
  if (e == cudaSuccess) e = cudaMemcpyAsync(hist, p.hist, sizeof(hist), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(parts.data(), p.partials, sizeof(double) * grid, cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(e, "diagnostics");
  for (int i = 0; i < kDiagShiftBins; ++i) out->displacement[i] = static_cast<int64_t>(hist[i]);
  for (int i = 0; i < kDiagMarginBins; ++i)
    out->margin[i] = static_cast<int64_t>(hist[kDiagShiftBins + i]);
  double sum = 0.0;
  for (int b = 0; b < grid; ++b) sum += parts[b];
  out->mean_max_prob = sum / static_cast<double>(sh.n);
  return GSQ_OK;
}

gsq_status gsq_project(gsq_layer* L, void* stream, uint8_t* codes_dev, float* margin_dev) {
  GSQ_INJECT("gsq_project");
  if (!valid(L)) return fail(GSQ_ERR_INVALID_ARG, "invalid layer handle");
  if (!codes_dev && !margin_dev) return GSQ_OK;
  DeviceGuard guard(L->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  ProjectParams p;
  p.n = L->shape.n;
  p.K = L->shape.L;
  p.nlev = L->shape.K;
  p.mask_sign = L->shape.mask_sign;
  p.j0 = L->shape.shift ? L->ws + L->lay.j0 : nullptr;
  p.logits = fptr(L, L->lay.logits);
  p.codes = codes_dev;
  p.margin = margin_dev;
  int slot;
  prof_begin(L, GSQ_K_PROJECT, s, slot);
  const cudaError_t e = launch_project(p, L->num_sms, s);
  prof_end(L, slot, s);
  if (e != cudaSuccess) return cuda_fail(e, "project kernel");
  return GSQ_OK;
}

gsq_status gsq_packed_size(const gsq_layer* L, size_t* bytes) {
  GSQ_INJECT("gsq_packed_size");
  if (!valid(L)) return fail(GSQ_ERR_INVALID_ARG, "invalid layer handle");
  if (!bytes) return fail(GSQ_ERR_INVALID_ARG, "bytes is NULL");
  *bytes = packed_bytes(L);
  return GSQ_OK;
}

gsq_status gsq_pack(gsq_layer* L, void* stream, void* out_dev, size_t cap, size_t* written) {
  GSQ_INJECT("gsq_pack");
  if (!valid(L)) return fail(GSQ_ERR_INVALID_ARG, "invalid layer handle");
  if (!out_dev) return fail(GSQ_ERR_INVALID_ARG, "out_dev is NULL");
  const size_t need = packed_bytes(L);
  if (cap < need) return fail(GSQ_ERR_INVALID_ARG, "pack buffer too small: %zu < %zu", cap, need);
  DeviceGuard guard(L->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  PackParams p;
  p.n = L->shape.n;
  p.K = L->shape.L;
  p.nlev = L->shape.K;
  p.mask_sign = L->shape.mask_sign;
  p.j0 = L->shape.shift ? L->ws + L->lay.j0 : nullptr;
  p.group = L->shape.group;
  p.kquant = L->shape.kquant;
  p.logits = fptr(L, L->lay.logits);
  p.scales = fptr(L, L->lay.scales);
  p.kq_d = L->shape.kquant ? reinterpret_cast<const uint16_t*>(L->ws + L->lay.kq_d) : nullptr;
  p.kq_sc = L->shape.kquant ? reinterpret_cast<const int8_t*>(L->ws + L->lay.kq_sc) : nullptr;
  p.out = static_cast<uint8_t*>(out_dev);
  p.code_bytes = static_cast<int64_t>(code_section_bytes(L->shape.n, L->shape.K));
  int slot;
  prof_begin(L, GSQ_K_PACK, s, slot);
  const cudaError_t e = launch_pack(p, L->num_sms, s);
  prof_end(L, slot, s);
  if (e != cudaSuccess) return cuda_fail(e, "pack kernel");
  if (written) *written = need;
  return GSQ_OK;
}

gsq_status gsq_tensor_size(const gsq_layer* L, int32_t which, size_t* bytes) {
  GSQ_INJECT("gsq_tensor_size");
  if (!valid(L)) return fail(GSQ_ERR_INVALID_ARG, "invalid layer handle");
  if (!bytes) return fail(GSQ_ERR_INVALID_ARG, "bytes is NULL");
  if (which < GSQ_T_LOGITS || which > GSQ_T_J0) return fail(GSQ_ERR_INVALID_ARG, "bad tensor id %d", which);
  *bytes = tensor_bytes(L, which);
  return GSQ_OK;
}

static gsq_status copy_tensor(gsq_layer* L, int32_t which, void* dst, const void* src, size_t bytes,
                              void* stream, const char* fn) {
  if (!valid(L)) return fail(GSQ_ERR_INVALID_ARG, "invalid layer handle");
  if (which < GSQ_T_LOGITS || which > GSQ_T_J0) return fail(GSQ_ERR_INVALID_ARG, "bad tensor id %d", which);
  const size_t need = tensor_bytes(L, which);
  if (need == 0) return fail(GSQ_ERR_INVALID_ARG, "%s: layer has no tensor %d", fn, which);
  if (bytes != need) return fail(GSQ_ERR_INVALID_ARG, "%s: bytes %zu != tensor size %zu", fn, bytes, need);
  if (!dst || !src) return fail(GSQ_ERR_INVALID_ARG, "%s: NULL buffer", fn);
  DeviceGuard guard(L->device);
  const cudaError_t e = cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDeviceToDevice, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, fn);
  return GSQ_OK;
}

gsq_status gsq_get_tensor(gsq_layer* L, int32_t which, void* dst_dev, size_t bytes, void* stream) {
  GSQ_INJECT("gsq_get_tensor");
  if (!valid(L)) return fail(GSQ_ERR_INVALID_ARG, "invalid layer handle");
  if (which == GSQ_T_G && !L->g_valid)
    return fail(GSQ_ERR_STATE, "G holds no step's gradient yet (no step has run)");
  return copy_tensor(L, which, dst_dev, L->ws + tensor_offset(L, which), bytes, stream, "gsq_get_tensor");
}

gsq_status gsq_set_tensor(gsq_layer* L, int32_t which, const void* src_dev, size_t bytes, void* stream) {
  GSQ_INJECT("gsq_set_tensor");
  if (!valid(L)) return fail(GSQ_ERR_INVALID_ARG, "invalid layer handle");
  const gsq_status st =
      copy_tensor(L, which, L->ws + tensor_offset(L, which), src_dev, bytes, stream, "gsq_set_tensor");
  if (st == GSQ_OK) L->d_ready = false;
  return st;
}

gsq_status gsq_sync_status(gsq_layer* L, void* stream) {
  GSQ_INJECT("gsq_sync_status");
  if (!valid(L)) return fail(GSQ_ERR_INVALID_ARG, "invalid layer handle");
  DeviceGuard guard(L->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  DevFlags* cflags = reinterpret_cast<DevFlags*>(L->ws + L->lay.flags);
  cudaError_t e = launch_canaries(L->ws, canary_list(L->lay), 0, cflags, s);
  if (e != cudaSuccess) return cuda_fail(e, "check canaries");
  e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(e, "gsq_sync_status");
  DevFlags* flags = reinterpret_cast<DevFlags*>(L->ws + L->lay.flags);
  unsigned int err = 0;
  e = cudaMemcpy(&err, &flags->error, sizeof(err), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e, "read error word");
  if (err) {
    cudaMemset(&flags->error, 0, sizeof(err));
    if ((err & 0xFFFF0000u) == kCanaryError) {
      const unsigned int i = err & 0xFFFFu;
      return fail(GSQ_ERR_STATE, "workspace canary after buffer '%s' was overwritten",
                  i < static_cast<unsigned int>(L->lay.ncanary) ? L->lay.canary_of[i] : "?");
    }
    return fail(GSQ_ERR_TIMEOUT, "a bounded device-side wait gave up (code 0x%x)", err);
  }
  return GSQ_OK;
}

gsq_status gsq_profile_enable(gsq_layer* L, int32_t on) {
  if (!valid(L)) return fail(GSQ_ERR_INVALID_ARG, "invalid layer handle");
  L->profiling = on != 0;
  return GSQ_OK;
}

gsq_status gsq_profile_read(gsq_layer* L, gsq_profile* out) {
  if (!valid(L)) return fail(GSQ_ERR_INVALID_ARG, "invalid layer handle");
  if (!out) return fail(GSQ_ERR_INVALID_ARG, "out is NULL");
  std::memset(out, 0, sizeof(*out));
  DeviceGuard guard(L->device);
  if (L->ev_used > 0) {
    cudaError_t e = cudaEventSynchronize(L->ev[2 * (L->ev_used - 1) + 1]);
    if (e != cudaSuccess) return cuda_fail(e, "profile sync");
    for (int i = 0; i < L->ev_used; ++i) {
      float ms = 0.f;
      e = cudaEventElapsedTime(&ms, L->ev[2 * i], L->ev[2 * i + 1]);
      if (e != cudaSuccess) return cuda_fail(e, "profile elapsed");
      out->launches[L->ev_kind[i]] += 1;
      out->total_ms[L->ev_kind[i]] += ms;
    }
  }
  L->ev_used = 0;
  return GSQ_OK;
}

gsq_status gsq_destroy(gsq_layer* L) {
  if (!valid(L)) return fail(GSQ_ERR_INVALID_ARG, "invalid layer handle");
  unregister_live(L);
  for (cudaEvent_t e : L->ev) cudaEventDestroy(e);
  L->magic = 0;
  delete L;
  return GSQ_OK;
}

const char* gsq_last_error(void) { return g_last_error.c_str(); }

const char* gsq_version(void) { return "0.2.0"; }

const char* gsq_kernel_name(gsq_layer* L, int32_t kind) {
  if (!valid(L)) return nullptr;
  if (kind == GSQ_K_GEMM) {
    if (!L->shape.d_bf16) return "k_simt_gemm";
    int mode = L->gemm_pair;
    if (mode == 1)
      mode = tc_gemm_cluster_mode(static_cast<int>(L->shape.E), static_cast<int>(L->shape.R),
                                  static_cast<int>(L->shape.C), L->tile_n, L->num_sms);
    return mode == 2 ? "k_tc_gemm_quad" : (mode ? "k_tc_gemm_pair" : "k_tc_gemm");
  }
  if (kind == GSQ_K_BACKWARD) {
    return L->grid_bwd_staged > 0 ? "k_backward_staged" : "k_backward";
  }
  return nullptr;
}

}  // extern "C"
