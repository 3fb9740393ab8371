"""ctypes binding of libgsq (include/gsq.h).

Argument marshalling only: every step of the quantizer runs in the library's
CUDA kernels.  The module-level functions carry the C names and raise GsqError
on a non-OK status; `Layer` owns a torch-allocated workspace and passes torch's
current CUDA stream.  PyTorch is used for device memory and streams only.

The library is loaded from this package directory (built by build.py); if it
is missing, importing this module fails loudly -- there is no CPU fallback.
"""
from __future__ import annotations

import ctypes
import os
from ctypes import (POINTER, Structure, byref, c_char_p, c_double, c_float, c_int32, c_int64,
                    c_size_t, c_uint32, c_uint64, c_void_p)
from typing import Optional, Sequence

# GSQ_LIBRARY, if set, names a libgsq.so built elsewhere (same ABI).
LIB_PATH = os.environ.get("GSQ_LIBRARY") or os.path.join(
    os.path.dirname(os.path.abspath(__file__)), "libgsq.so")

# ---- constants mirrored from gsq.h -------------------------------------------
GSQ_OK, GSQ_ERR_INVALID_ARG, GSQ_ERR_SHAPE, GSQ_ERR_WORKSPACE, GSQ_ERR_CUDA = 0, 1, 2, 3, 4
GSQ_ERR_NONFINITE, GSQ_ERR_STATE, GSQ_ERR_TIMEOUT, GSQ_ERR_INJECTED, GSQ_ERR_UNSUPPORTED = 5, 6, 7, 8, 9
GSQ_MAX_LEVELS = 8
GSQ_DTYPE_F32, GSQ_DTYPE_BF16 = 0, 1
GSQ_CALIB_H, GSQ_CALIB_X, GSQ_CALIB_BATCHES = 0, 1, 2
GSQ_SCALE_GROUP, GSQ_SCALE_KQUANT2 = 0, 1
GSQ_GEMM_BF16, GSQ_GEMM_F32 = 0, 1
GSQ_FLAG_NO_NOISE, GSQ_FLAG_UNSTAGED = 1, 8
GSQ_PARAM_FULL, GSQ_PARAM_SHIFT5, GSQ_PARAM_MASK_SIGN = 0, 1, 2
PARAM_MODES = {"full": GSQ_PARAM_FULL, "shift5": GSQ_PARAM_SHIFT5, "mask_sign": GSQ_PARAM_MASK_SIGN}
(GSQ_T_LOGITS, GSQ_T_SCALES, GSQ_T_MOM_LOGITS, GSQ_T_MOM_SCALES, GSQ_T_D, GSQ_T_G, GSQ_T_W,
 GSQ_T_H, GSQ_T_KQ_D, GSQ_T_KQ_SC, GSQ_T_J0) = range(11)
(GSQ_K_FORWARD, GSQ_K_GEMM, GSQ_K_BACKWARD, GSQ_K_PROJECT, GSQ_K_PACK, GSQ_K_INIT,
 GSQ_K_TOKENS) = range(7)
GSQ_K_COUNT = 7
KERNEL_NAMES = ["forward", "gemm", "backward", "project", "pack", "init", "tokens"]

EXPORTED = ["gsq_workspace_size", "gsq_init_layer", "gsq_step", "gsq_forward", "gsq_project",
            "gsq_packed_size", "gsq_pack", "gsq_tensor_size", "gsq_get_tensor", "gsq_set_tensor",
            "gsq_sync_status", "gsq_profile_enable", "gsq_profile_read", "gsq_destroy",
            "gsq_last_error", "gsq_version", "gsq_backward_update_noalloc", "gsq_init_logits",
            "gsq_step_tokens", "gsq_diagnose", "gsq_kernel_name"]


GSQ_DIAG_SHIFT_BINS, GSQ_DIAG_MARGIN_BINS = 8, 9


class gsq_diagnostics(Structure):
    _fields_ = [("displacement", c_int64 * GSQ_DIAG_SHIFT_BINS),
                ("margin", c_int64 * GSQ_DIAG_MARGIN_BINS), ("mean_max_prob", c_double)]


class gsq_layer_desc(Structure):
    _fields_ = [
        ("num_experts", c_int32), ("out_features", c_int32), ("in_features", c_int32),
        ("w_dtype", c_int32), ("W", c_void_p), ("calib", c_void_p), ("n_tokens", c_int64),
        ("calib_kind", c_int32), ("num_levels", c_int32), ("grid", c_float * GSQ_MAX_LEVELS),
        ("group_size", c_int32), ("scale_mode", c_int32), ("init_bias", c_float),
        ("flags", c_uint32), ("seed", c_uint64), ("lr_logits", c_float), ("lr_scales", c_float),
        ("beta1", c_float), ("beta2", c_float), ("wd_logits", c_float), ("wd_scales", c_float),
        ("gemm_precision", c_int32), ("param_mode", c_int32), ("index_offset", c_uint64),
    ]


class gsq_profile(Structure):
    _fields_ = [("launches", c_int32 * GSQ_K_COUNT), ("total_ms", c_float * GSQ_K_COUNT)]


class gsq_backward_args(Structure):
    _fields_ = [
        ("num_experts", c_int32), ("out_features", c_int32), ("in_features", c_int32),
        ("num_levels", c_int32), ("grid", c_float * GSQ_MAX_LEVELS), ("group_size", c_int32),
        ("w_dtype", c_int32), ("d_dtype", c_int32), ("flags", c_uint32), ("W", c_void_p),
        ("G", c_void_p), ("logits", c_void_p), ("m_logits", c_void_p), ("scales", c_void_p),
        ("m_scales", c_void_p), ("loss_dev", c_void_p), ("seed", c_uint64), ("step", c_uint64),
        ("tau", c_float), ("kappa", c_float), ("lr_logits", c_float), ("lr_scales", c_float),
        ("beta1", c_float), ("beta2", c_float), ("wd_logits", c_float), ("wd_scales", c_float),
    ]


class GsqError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"gsq status {status}: {message}")
        self.status = status


def load_library(path: str = LIB_PATH) -> ctypes.CDLL:
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is not built; run `python -c 'import __graft_entry__ as g; g.build()'`")
    lib = ctypes.CDLL(path)
    P = c_void_p
    sig = {
        "gsq_workspace_size": (c_int32, [POINTER(gsq_layer_desc), POINTER(c_size_t)]),
        "gsq_init_layer": (c_int32, [POINTER(gsq_layer_desc), P, c_size_t, P, POINTER(c_void_p)]),
        "gsq_step": (c_int32, [P, c_uint64, c_float, c_float, c_float, c_float, P, P, P, P]),
        "gsq_forward": (c_int32, [P, c_uint64, c_float, c_float, P, P]),
        "gsq_project": (c_int32, [P, P, P, P]),
        "gsq_packed_size": (c_int32, [P, POINTER(c_size_t)]),
        "gsq_pack": (c_int32, [P, P, P, c_size_t, POINTER(c_size_t)]),
        "gsq_tensor_size": (c_int32, [P, c_int32, POINTER(c_size_t)]),
        "gsq_get_tensor": (c_int32, [P, c_int32, P, c_size_t, P]),
        "gsq_set_tensor": (c_int32, [P, c_int32, P, c_size_t, P]),
        "gsq_sync_status": (c_int32, [P, P]),
        "gsq_profile_enable": (c_int32, [P, c_int32]),
        "gsq_profile_read": (c_int32, [P, POINTER(gsq_profile)]),
        "gsq_destroy": (c_int32, [P]),
        "gsq_last_error": (c_char_p, []),
        "gsq_version": (c_char_p, []),
        "gsq_kernel_name": (c_char_p, [P, c_int32]),
        "gsq_backward_update_noalloc": (c_int32, [POINTER(gsq_backward_args), P]),
        "gsq_init_logits": (c_int32, [P, P, P, c_float, c_float, P]),
        "gsq_diagnose": (c_int32, [P, c_float, c_float, P, POINTER(gsq_diagnostics)]),
        "gsq_step_tokens": (c_int32, [P, c_uint64, c_uint32, c_uint32, c_float, c_float, c_float,
                                      c_float, P, c_int64, P, P]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


_lib = load_library()


def _check(status: int) -> None:
    if status != GSQ_OK:
        raise GsqError(status, _lib.gsq_last_error().decode())


def _ptr(t) -> Optional[int]:
    return None if t is None else int(t.data_ptr())


# ---- the C entry points, same names -----------------------------------------
def gsq_workspace_size(desc: gsq_layer_desc) -> int:
    out = c_size_t(0)
    _check(_lib.gsq_workspace_size(byref(desc), byref(out)))
    return out.value


def gsq_init_layer(desc: gsq_layer_desc, workspace_ptr: int, nbytes: int, stream: int) -> int:
    handle = c_void_p(0)
    _check(_lib.gsq_init_layer(byref(desc), workspace_ptr, nbytes, stream, byref(handle)))
    return handle.value


def gsq_step(handle: int, step: int, tau: float, kappa: float, next_tau: float, next_kappa: float,
             stream: int, loss_ptr=None, grad_logits_ptr=None, grad_scales_ptr=None) -> None:
    _check(_lib.gsq_step(handle, step, tau, kappa, next_tau, next_kappa, stream, loss_ptr,
                         grad_logits_ptr, grad_scales_ptr))


def gsq_forward(handle: int, step: int, tau: float, kappa: float, stream: int, what_ptr=None) -> None:
    _check(_lib.gsq_forward(handle, step, tau, kappa, stream, what_ptr))


def gsq_step_tokens(handle: int, step: int, micro: int, n_micro: int, tau: float, kappa: float,
                    next_tau: float, next_kappa: float, X_ptr, n_tokens: int, stream: int,
                    loss_ptr=None) -> None:
    _check(_lib.gsq_step_tokens(handle, step, micro, n_micro, tau, kappa, next_tau, next_kappa,
                                X_ptr, n_tokens, stream, loss_ptr))


def gsq_diagnose(handle: int, tau: float, kappa: float, stream: int) -> dict:
    out = gsq_diagnostics()
    _check(_lib.gsq_diagnose(handle, tau, kappa, stream, byref(out)))
    return {"displacement": list(out.displacement), "margin": list(out.margin),
            "mean_max_prob": out.mean_max_prob}


def gsq_init_logits(handle: int, codes_ptr, eps_ptr, alpha: float, sigma: float, stream: int) -> None:
    _check(_lib.gsq_init_logits(handle, codes_ptr, eps_ptr, alpha, sigma, stream))


def gsq_project(handle: int, stream: int, codes_ptr=None, margin_ptr=None) -> None:
    _check(_lib.gsq_project(handle, stream, codes_ptr, margin_ptr))


def gsq_packed_size(handle: int) -> int:
    out = c_size_t(0)
    _check(_lib.gsq_packed_size(handle, byref(out)))
    return out.value


def gsq_pack(handle: int, stream: int, out_ptr: int, cap: int) -> int:
    written = c_size_t(0)
    _check(_lib.gsq_pack(handle, stream, out_ptr, cap, byref(written)))
    return written.value


def gsq_tensor_size(handle: int, which: int) -> int:
    out = c_size_t(0)
    _check(_lib.gsq_tensor_size(handle, which, byref(out)))
    return out.value


def gsq_get_tensor(handle: int, which: int, dst_ptr: int, nbytes: int, stream: int) -> None:
    _check(_lib.gsq_get_tensor(handle, which, dst_ptr, nbytes, stream))


def gsq_set_tensor(handle: int, which: int, src_ptr: int, nbytes: int, stream: int) -> None:
    _check(_lib.gsq_set_tensor(handle, which, src_ptr, nbytes, stream))


def gsq_sync_status(handle: int, stream: int) -> None:
    _check(_lib.gsq_sync_status(handle, stream))


def gsq_profile_enable(handle: int, on: bool) -> None:
    _check(_lib.gsq_profile_enable(handle, 1 if on else 0))


def gsq_profile_read(handle: int) -> dict:
    prof = gsq_profile()
    _check(_lib.gsq_profile_read(handle, byref(prof)))
    return {KERNEL_NAMES[k]: (prof.launches[k], prof.total_ms[k]) for k in range(GSQ_K_COUNT)}


def gsq_destroy(handle: int) -> None:
    _check(_lib.gsq_destroy(handle))


def gsq_last_error() -> str:
    return _lib.gsq_last_error().decode()


def gsq_version() -> str:
    return _lib.gsq_version().decode()


def gsq_kernel_name(handle, kind: int):
    """The kernel gsq_step launches for GSQ_K_GEMM or GSQ_K_BACKWARD, or None."""
    r = _lib.gsq_kernel_name(handle, kind)
    return None if r is None else r.decode()


def gsq_backward_update_noalloc(args: gsq_backward_args, stream: int) -> None:
    """The allocation-free backward + Lion update (see include/gsq.h)."""
    _check(_lib.gsq_backward_update_noalloc(byref(args), stream))


# ---- convenience wrapper over torch memory and streams -----------------------
def make_desc(*, experts: int, rows: int, cols: int, grid: Sequence[float], group_size: int,
              w_dtype: int = GSQ_DTYPE_BF16, W_ptr: int = 0, calib_ptr: int = 0,
              calib_kind: int = GSQ_CALIB_H, n_tokens: int = 0, scale_mode: int = GSQ_SCALE_GROUP,
              init_bias: float = 2.0, seed: int = 0, lr_logits: float = 1e-4,
              lr_scales: float = 5e-5, beta1: float = 0.9, beta2: float = 0.95,
              wd_logits: float = 1.0, wd_scales: float = 0.0, gemm: int = GSQ_GEMM_BF16,
              noise: bool = True, param_mode: int = GSQ_PARAM_FULL,
              unstaged: bool = False, index_offset: int = 0) -> gsq_layer_desc:
    d = gsq_layer_desc()
    d.num_experts, d.out_features, d.in_features = experts, rows, cols
    d.w_dtype = w_dtype
    d.W, d.calib = W_ptr, calib_ptr
    d.n_tokens = n_tokens
    d.calib_kind = calib_kind
    d.num_levels = len(grid)
    for k, q in enumerate(list(grid)[:GSQ_MAX_LEVELS]):
        d.grid[k] = q
    d.group_size = group_size
    d.scale_mode = scale_mode
    d.init_bias = init_bias
    d.flags = (0 if noise else GSQ_FLAG_NO_NOISE) | (GSQ_FLAG_UNSTAGED if unstaged else 0)
    d.seed = seed
    d.lr_logits, d.lr_scales = lr_logits, lr_scales
    d.beta1, d.beta2 = beta1, beta2
    d.wd_logits, d.wd_scales = wd_logits, wd_scales
    d.gemm_precision = gemm
    d.param_mode = param_mode
    d.index_offset = index_offset
    return d


class Layer:
    """One layer problem on the current CUDA device.

    W: [E, R, C] (fp32 or bf16, CUDA); calib: H [E, C, C] or X [E, T, C] fp32
    (CUDA).  The workspace is a torch uint8 tensor owned by this object."""

    def __init__(self, W, calib, grid: Sequence[float], group_size: int, *, calib_kind: str = "H",
                 scale_mode: str = "group", gemm: str = "bf16", param: str = "full", stream=None,
                 tokens_per_batch: int = 0, **hyper):
        """calib_kind "batches": no calibration at init (calib may be None); every
        micro-batch brings up to tokens_per_batch tokens through step_tokens."""
        import torch
        self._torch = torch
        batches = calib_kind == "batches"
        assert W.is_cuda and W.dim() == 3
        if not batches:
            assert calib is not None and calib.is_cuda and calib.dim() == 3
            calib = calib.contiguous().float()
        W = W.contiguous()
        E, R, C = W.shape
        self.shape = (E, R, C)
        self.K = len(grid)
        if param not in PARAM_MODES:
            raise ValueError(f"param must be one of {sorted(PARAM_MODES)}")
        self.L = {"full": self.K, "shift5": 5, "mask_sign": 2}[param]   # logits per weight
        self.group_size = group_size
        self.desc = make_desc(
            experts=E, rows=R, cols=C, grid=grid, group_size=group_size,
            w_dtype=GSQ_DTYPE_BF16 if W.dtype == torch.bfloat16 else GSQ_DTYPE_F32,
            W_ptr=_ptr(W), calib_ptr=_ptr(calib) if not batches else 0,
            calib_kind={"X": GSQ_CALIB_X, "batches": GSQ_CALIB_BATCHES}.get(calib_kind, GSQ_CALIB_H),
            n_tokens=calib.shape[1] if calib_kind == "X" else (tokens_per_batch if batches else 0),
            scale_mode=GSQ_SCALE_KQUANT2 if scale_mode == "kquant2" else GSQ_SCALE_GROUP,
            gemm=GSQ_GEMM_F32 if gemm == "f32" else GSQ_GEMM_BF16,
            param_mode=PARAM_MODES[param], **hyper)
        if W.dtype not in (torch.float32, torch.bfloat16):
            raise TypeError("W must be fp32 or bf16")
        nbytes = gsq_workspace_size(self.desc)
        self.workspace = torch.empty(nbytes, dtype=torch.uint8, device=W.device)
        self.stream = stream
        self.handle = gsq_init_layer(self.desc, _ptr(self.workspace), nbytes, self._stream())
        self.desc.W = None
        self.desc.calib = None

    def _stream(self) -> int:
        s = self.stream if self.stream is not None else self._torch.cuda.current_stream()
        return int(s.cuda_stream)

    def step(self, t: int, tau: float, kappa: float = 1.0, next_tau: float = 0.0,
             next_kappa: float = 1.0, loss=None, grad_logits=None, grad_scales=None) -> None:
        gsq_step(self.handle, t, tau, kappa, next_tau, next_kappa, self._stream(), _ptr(loss),
                 _ptr(grad_logits), _ptr(grad_scales))

    def step_tokens(self, step: int, micro: int, n_micro: int, tau: float, X, kappa: float = 1.0,
                    next_tau: float = 0.0, next_kappa: float = 1.0, loss=None) -> None:
        """One micro-batch (tokens X: fp32 [E, T, C] on the device) of a step with
        gradient accumulation; the update follows the last micro-batch."""
        X = X.contiguous()
        gsq_step_tokens(self.handle, step, micro, n_micro, tau, kappa, next_tau, next_kappa,
                        _ptr(X), X.shape[1], self._stream(), _ptr(loss))

    def forward(self, t: int, tau: float, kappa: float = 1.0, what=None) -> None:
        gsq_forward(self.handle, t, tau, kappa, self._stream(), _ptr(what))

    def init_logits(self, codes, eps=None, alpha: float = 1.0, sigma: float = 1.0) -> None:
        """Warm start from supplied codes (uint8 [E, R, C]) and optional eps ([L, E, R, C] fp32)."""
        codes = codes.contiguous()
        eps = None if eps is None else eps.contiguous()
        gsq_init_logits(self.handle, _ptr(codes), _ptr(eps), alpha, sigma, self._stream())

    def kernel_name(self, kind: int):
        """Kernel gsq_step launches for GSQ_K_GEMM or GSQ_K_BACKWARD on this layer."""
        return gsq_kernel_name(self.handle, kind)

    def diagnose(self, tau: float, kappa: float = 1.0) -> dict:
        """Displacement and margin histograms and the mean max-probability (see gsq.h)."""
        return gsq_diagnose(self.handle, tau, kappa, self._stream())

    def project(self, codes=None, margin=None) -> None:
        gsq_project(self.handle, self._stream(), _ptr(codes), _ptr(margin))

    def packed_size(self) -> int:
        return gsq_packed_size(self.handle)

    def pack(self, out) -> int:
        return gsq_pack(self.handle, self._stream(), _ptr(out), out.numel() * out.element_size())

    def tensor_size(self, which: int) -> int:
        return gsq_tensor_size(self.handle, which)

    def get_tensor(self, which: int, dtype=None):
        torch = self._torch
        nbytes = self.tensor_size(which)
        out = torch.empty(nbytes, dtype=torch.uint8, device=self.workspace.device)
        gsq_get_tensor(self.handle, which, _ptr(out), nbytes, self._stream())
        return out.view(dtype) if dtype is not None else out

    def set_tensor(self, which: int, src) -> None:
        src = src.contiguous()
        gsq_set_tensor(self.handle, which, _ptr(src), src.numel() * src.element_size(),
                       self._stream())

    def sync_status(self) -> None:
        gsq_sync_status(self.handle, self._stream())

    def profile_enable(self, on: bool = True) -> None:
        gsq_profile_enable(self.handle, on)

    def profile_read(self) -> dict:
        return gsq_profile_read(self.handle)

    def close(self) -> None:
        if getattr(self, "handle", None):
            gsq_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
