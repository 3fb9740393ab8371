// Internal declarations shared by the libgsq CUDA sources (not part of the ABI).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/gsq.h"

namespace gsq {

constexpr int kMaxLevels = GSQ_MAX_LEVELS;
constexpr int kSubBlock = 16;     // K-Quant-like sub-block (6-bit sub-scale)
constexpr int kSuperBlock = 256;  // K-Quant-like super-block (fp16 d)
constexpr int kKqRecord = 110;    // bytes per packed super-block
constexpr int kEwThreads = 256;   // threads per block of the elementwise kernels

// Programmatic dependent launch. A kernel launched with the programmatic stream
// serialization attribute (set by pdl_attr) may be scheduled while the kernel before it on
// the stream is still running; grid_dep_wait() returns once that kernel has completed and
// its writes are visible, so it comes before every access to global memory the kernel
// before may read or write. grid_dep_launch() lets the next such kernel be scheduled onto
// SMs this one frees. Without the attribute both are no-ops (PTX griddepcontrol, sm_90+).
#ifdef __CUDACC__
__device__ __forceinline__ void grid_dep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void grid_dep_launch() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
#endif
inline void pdl_attr(cudaLaunchAttribute& a) {
  a.id = cudaLaunchAttributeProgrammaticStreamSerialization;
  a.val.programmaticStreamSerializationAllowed = 1;
}

// Device-side status words, one 256-byte slot of the workspace.
struct DevFlags {
  unsigned int blocks_done;  // last-block-done counter of the loss reduction
  unsigned int error;        // nonzero: a bounded wait gave up (code of the site)
  unsigned int nonfinite;    // init scan: count of non-finite inputs
  unsigned int pad[61];
};

// Philox4x32-10 round keys: k0[r] = key0 + r * 0x9E3779B9, k1[r] = key1 + r * 0xBB67AE85.
struct PhiloxRoundKeys {
  uint32_t k0[10], k1[10];
};

// Everything the elementwise kernels need, passed by value.
struct EwParams {
  // shape
  int64_t n;          // E*R*C weights
  int64_t nq;         // n / 4 quads
  int K;              // logits per weight: grid levels, 5 shifts, or 2 (mask, sign)
  int nlev;           // grid levels
  int mode;           // GSQ_PARAM_FULL / GSQ_PARAM_SHIFT5 / GSQ_PARAM_MASK_SIGN
  const uint8_t* j0;  // local shift: initial grid index per weight [n]; null otherwise
  int group;          // scale group (16 for K-Quant)
  int log2_group;
  int w_bf16;         // W storage: 1 bf16, 0 fp32
  int d_bf16;         // D storage: 1 bf16, 0 fp32
  float grid[kMaxLevels];
  // state (device)
  float* logits;      // [K][n]
  float* m_logits;    // [K][n]
  float* scales;      // [n/group]
  float* m_scales;    // [n/group]
  const void* W;      // [n]
  void* D;            // [n]
  const float* G;     // [n]
  // noise
  PhiloxRoundKeys keys;
  int noise;          // 0: g = 0
  uint64_t index_base;  // noise counter index of weight 0 (a shard's offset in the whole layer)
  // step t (backward / forward)
  uint32_t t;
  float kappa_log2, inv_tau, kappa_over_tau;  // kappa_log2 = kappa * log2(e)
  // look-ahead forward (t + 1)
  int lookahead;
  uint32_t t_next;
  float kappa_log2_next, inv_tau_next;
  // Lion
  float lr_l, lr_s, b1, b2, wd_l, wd_s;
  float lrwd_l, lrwd_s;  // lr * wd, rounded once from double
  int scales_frozen;
  // outputs
  float* grad_logits;  // export mode: [K][n]
  float* grad_scales;  // export mode: [n/group]
  // gradient accumulation over micro-batches: when set, every gradient becomes
  // (this pass's + acc_in) * acc_scale before export or the Lion update
  const float* acc_in_l;  // [K][n] or null
  const float* acc_in_s;  // [n/group] or null
  float acc_scale;
  float* what;         // forward: optional W^ export [n]
  double* loss_partials;
  DevFlags* flags;
  float* loss_out;     // nullable
  int stall;           // test hook (GSQ_TEST_STALL=backward): the staged backward never fills
                       // its second stage, so a bounded wait runs out and reports 0x7C03
};

// Byte offsets of one stage's streams in the staged backward's shared memory
// (a tile of 1,024 weights); bytes = stage size, tx = bytes the copies deliver.
struct BwdStage {
  uint32_t l, m, g, w, s, ms, j, bytes, tx;
};

// Records `msg` as this thread's gsq_last_error() text and returns `st` (gsq_api.cu).
gsq_status set_last_error(gsq_status st, const char* msg);

// ---- launchers (gsq_elementwise.cu; backward: gsq_backward.cu, gsq_staged.cu) --
cudaError_t launch_forward(const EwParams& p, int grid, cudaStream_t s);
// pdl: launched with pdl_attr (the kernels wait for the one before them first).
cudaError_t launch_backward(const EwParams& p, int grid, cudaStream_t s, bool pdl = false);
// TMA-staged backward for non-export, non-accumulating steps: its grid for a
// layer (resident blocks x SMs) and staging plan, 0 where it does not apply;
// and its launch.
int ew_staged_grid(int K, int mode, int w_bf16, int log2_group, int scales_frozen, int num_sms,
                   int* plan);
cudaError_t launch_backward_staged(const EwParams& p, int grid, int plan, cudaStream_t s,
                                   bool pdl = false);
int ew_grid_size(int K, int which, int num_sms, int mode);  // which: 0 forward, 1 backward
int ew_backward_grid(int K, int num_sms, int mode);          // gsq_backward.cu

struct InitParams {
  int64_t n;
  int K;               // grid levels
  int mask_sign;       // logits are the (mask, sign) planes, Eq. 3 from the RTN code
  uint8_t* j0;         // local shift: receives the RTN index; logits then hold 5 planes
  uint8_t* code0;      // receives the initial grid code of every weight (diagnostics)
  int group;
  int kquant;
  int w_bf16;
  float grid[kMaxLevels];
  float init_bias;
  const void* W;       // stored copy
  float* logits;
  float* m_logits;
  float* scales;
  float* m_scales;
  uint16_t* kq_d;      // [n/256]
  int8_t* kq_sc;       // [n/16]
};
cudaError_t launch_init_state(const InitParams& p, int num_sms, cudaStream_t s);

// Workspace canaries: 256 bytes after every buffer, written with a fixed word at
// init and checked later; a mismatch stores kCanaryError | index in flags->error.
constexpr int kMaxCanaries = 32;
constexpr unsigned int kCanaryError = 0xCA000000u;
struct CanaryList {
  int count;
  uint64_t off[kMaxCanaries];
};
cudaError_t launch_canaries(uint8_t* ws, const CanaryList& list, int write, DevFlags* flags,
                            cudaStream_t s);

struct InitCodesParams {
  int64_t n;
  int K;               // grid levels
  int mode;            // GSQ_PARAM_*
  float grid[kMaxLevels];
  const uint8_t* codes;
  const float* eps;    // [L][n] or null
  float alpha, sigma;
  float* logits;       // [L][n]
  float* m_logits;     // [L][n]
  uint8_t* j0;         // local shift: receives the codes
  uint8_t* code0;      // receives the codes (initial codes for the diagnostics)
};
cudaError_t launch_init_from_codes(const InitCodesParams& p, int num_sms, cudaStream_t s);
cudaError_t launch_nonfinite_scan(const void* x, int64_t count, int is_bf16,
                                  unsigned int* counter, cudaStream_t s);

struct ProjectParams {
  int64_t n;
  int K;               // logits per weight
  int nlev;            // grid levels
  int mask_sign;       // code from the hard rule l >= 0 of the mask and sign logits
  const uint8_t* j0;   // local shift (null otherwise): code = clip(j0 + argmax - 2)
  const float* logits;
  uint8_t* codes;
  float* margin;
};
cudaError_t launch_project(const ProjectParams& p, int num_sms, cudaStream_t s);

constexpr int kDiagShiftBins = 8;   // |code - initial code| = 0..6, >= 7
constexpr int kDiagMarginBins = 9;  // margins split at 1e-6, 1e-5, ..., 1, 10
struct DiagParams {
  int64_t n;
  int K;               // logits per weight
  int nlev;            // grid levels
  int mask_sign;
  const uint8_t* j0;   // local shift (null otherwise)
  const float* logits;
  const uint8_t* code0;
  double kappa_over_tau;
  unsigned long long* hist;  // [kDiagShiftBins + kDiagMarginBins], zeroed by the caller
  double* partials;          // [grid] sums of the max probability
};
cudaError_t launch_diagnose(const DiagParams& p, int grid, cudaStream_t s);

struct PackParams {
  int64_t n;
  int K;               // logits per weight
  int nlev;            // grid levels (code width)
  int mask_sign;       // code from the hard rule l >= 0 of the mask and sign logits
  const uint8_t* j0;   // local shift (null otherwise)
  int group;
  int kquant;
  const float* logits;
  const float* scales;     // group mode
  const uint16_t* kq_d;    // kquant
  const int8_t* kq_sc;     // kquant
  uint8_t* out;
  int64_t code_bytes;      // group mode: size of the padded code section
};
cudaError_t launch_pack(const PackParams& p, int num_sms, cudaStream_t s);

// ---- GEMMs (gsq_gemm_simt.cu, gsq_gemm_tc.cu) --------------------------------
// C[b][m][n] = alpha * sum_k A[b][m*sam + k*sak] * B[b][k*sbk + n*sbn]
struct SimtGemm {
  int batch, M, N, Kd;
  const void* A;
  int64_t sam, sak, sab;
  const void* B;
  int64_t sbk, sbn, sbb;
  float* C;
  int64_t ldc, scb;
  float alpha;
  int bf16_inputs;  // 1: A and B are bf16, else fp32
};
cudaError_t launch_simt_gemm(const SimtGemm& g, cudaStream_t s);

// H_out[e] = (H[e] + H[e]^T) / 2 converted to bf16 (out_bf16=1) or fp32.
cudaError_t launch_symmetrize(const float* H, void* out, int E, int C, int out_bf16,
                              cudaStream_t s);
// H[e][i][j] = H[e][j][i] for i > j, bf16 [E][C][C] in place (the lower triangle of a
// symmetric output whose upper triangle a TcGemm with sym = 1 computed).
cudaError_t launch_mirror_upper_bf16(void* H, int E, int C, cudaStream_t s);
// Xb[e] = bf16(X[e]) ([T][C]) and Xt[e] = bf16(X[e])^T ([C][ldt], first T columns);
// Xb null: Xt alone (ldt a multiple of 8).
cudaError_t launch_tokens_bf16(const float* X, void* Xb, void* Xt, int E, int T, int C, int ldt,
                               cudaStream_t s);

// tcgen05 / TMA bf16 GEMM: G[e] = alpha * D[e] (R x C, bf16, row-major) *
// H[e]^T (C x C, bf16, row-major; symmetric so H^T = H), fp32 out.
// out[e][m][n] = alpha * sum_k A[e][m][k] * B[e][n][k], bf16 operands (both
// K-major, rows of K elements), fp32 accumulation, fp32 or bf16 output.
// Needs K % 8 == 0 and N % 4 == 0.
struct TcGemm {
  int E, M, N, K;
  const void* A;   // [E*M][K] bf16
  const void* B;   // [E*N][K] bf16
  void* out;       // [E][M][N]
  int out_bf16;
  float alpha;
  DevFlags* flags;
  int tile_n;   // 0: choose 128 or 256 by wave balance
  int group_n;  // tile-order column group; <= 0: one group (m fastest across all columns)
  int pair;     // 0: single CTAs; 3: CTA pairs (cta_group::2, 256-row tiles over two SMs);
                // 2: clusters of two pairs sharing B by multicast; 1: pairs or clusters of
                // pairs, whichever tc_gemm_cluster_mode picks for the shape
  int stall;    // test hook (GSQ_TEST_STALL=gemm): the first k-block is never loaded
  int pdl;      // 1: tensor-core kernels launched with pdl_attr (prologue overlaps the
                // previous kernel's tail; operands read after grid_dep_wait)
  int sym;      // 1: symmetric output (M = N, out = A A^T with B = A): only the tiles
                // of the upper triangle are computed; launch_mirror_upper_bf16 fills
                // the rest (clusters of pairs fall back to pairs)
};
bool tc_gemm_supported(int device);

int tc_gemm_tile_n(int E, int M, int N, int num_sms, int pair);
// 2 (clusters of two CTA pairs) or 3 (CTA pairs) for an E x M x N contraction with
// tiles BN wide: clusters unless their resident count costs more than 6% more waves.
int tc_gemm_cluster_mode(int E, int M, int N, int bn, int num_sms);
cudaError_t launch_tc_gemm(const TcGemm& g, int num_sms, cudaStream_t s);

}  // namespace gsq
