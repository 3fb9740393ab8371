"""C-ABI checks that need no GPU: the library loads and exports every function
include/gsq.h declares; the ctypes descriptor matches the C layout (checked by
compiling the header with gcc); host-side validation, workspace sizing and
fault injection answer before any CUDA call."""
import ctypes
import os
import re
import subprocess
import sys
import textwrap

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "gsq.h")


@pytest.fixture(scope="module")
def lib():
    sys.path.insert(0, ROOT)
    from paper_2604_18556_gb300 import build
    build.build()
    from paper_2604_18556_gb300 import gsq
    return gsq


def _declared():
    src = open(HEADER).read()
    return sorted(set(re.findall(r"GSQ_API\s+[\w\s\*]+?\b(gsq_\w+)\s*\(", src)))


def test_every_declared_symbol_is_exported(lib):
    names = _declared()
    assert len(names) >= 16
    out = subprocess.run(["nm", "-D", "--defined-only", lib.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    exported = {ln.split()[-1] for ln in out.splitlines() if ln.strip()}
    assert set(names) <= exported
    assert set(names) == set(lib.EXPORTED)
    # the statically linked CUDA runtime stays private
    assert not any(s.startswith("cuda") for s in exported)
    cdll = ctypes.CDLL(lib.LIB_PATH)
    for n in names:
        assert getattr(cdll, n) is not None


@pytest.mark.parametrize("struct", ["gsq_layer_desc", "gsq_profile", "gsq_backward_args",
                                    "gsq_diagnostics"])
def test_struct_layout_matches_c(lib, tmp_path, struct):
    cls = getattr(lib, struct)
    fields = [f for f, _ in cls._fields_]
    prog = "#include <stdio.h>\n#include <stddef.h>\n#include \"gsq.h\"\nint main(void){\n"
    prog += f'printf("size %zu\\n", sizeof({struct}));\n'
    for f in fields:
        prog += f'printf("{f} %zu\\n", offsetof({struct}, {f}));\n'
    prog += "return 0;}\n"
    c = tmp_path / "layout.c"
    c.write_text(prog)
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-I", os.path.join(ROOT, "include"), str(c), "-o", str(exe)], check=True)
    out = dict(ln.split() for ln in subprocess.run([str(exe)], capture_output=True, text=True,
                                                   check=True).stdout.splitlines())
    assert int(out["size"]) == ctypes.sizeof(cls)
    for f in fields:
        assert int(out[f]) == getattr(cls, f).offset, f


def _desc(lib, **kw):
    base = dict(experts=1, rows=64, cols=256, grid=(-1.5, -0.5, 0.5, 1.5), group_size=128)
    base.update(kw)
    return lib.make_desc(**base)


def _align(x):
    return (x + 255) // 256 * 256


def test_workspace_size_formula(lib):
    from paper_2604_18556_gb300.configs import WORKLOADS
    for w in WORKLOADS.values():
        d = lib.make_desc(experts=w.experts, rows=w.rows, cols=w.cols, grid=w.grid,
                          group_size=w.group, w_dtype=lib.GSQ_DTYPE_F32 if w.w_dtype == "f32" else lib.GSQ_DTYPE_BF16,
                          calib_kind={"X": lib.GSQ_CALIB_X, "batches": lib.GSQ_CALIB_BATCHES}.get(
                              w.calib, lib.GSQ_CALIB_H),
                          n_tokens=w.tokens if w.calib in ("X", "batches") else 0,
                          scale_mode=lib.GSQ_SCALE_KQUANT2 if w.scale_mode == "kquant2" else lib.GSQ_SCALE_GROUP,
                          lr_scales=w.lr_scales,
                          param_mode=lib.PARAM_MODES[w.param])
        n, L = w.n, w.L
        # per-step tokens contract through each micro-batch's Gram matrix X^T X (formed from
        # its upper triangle) where that costs fewer flops than Y = D X^T, G = 2 Y X:
        # C (T + 2R) < 4 R T
        gram = w.calib == "batches" and w.cols * (w.tokens + 2 * w.rows) < 4 * w.rows * w.tokens
        # every buffer is 256-byte aligned and followed by a 256-byte canary
        bufs = [256, 8 * 16384, 4 * L * n, 4 * L * n, 4 * n // w.group, 4 * n // w.group,
                n * w.w_bytes()]
        if w.calib != "batches" or gram:
            bufs.append(w.experts * w.cols ** 2 * 2)               # H (bf16)
        bufs.append(2 * n)                                         # D (bf16)
        if w.calib != "batches":
            bufs.append(2 * n)                                     # D of the odd steps
        bufs.append(4 * n)                                         # G
        if w.scale_mode == "kquant2":
            bufs += [2 * n // 256, n // 16]
        if w.calib == "X":
            bufs.append(4 * w.experts * w.cols ** 2)
        if w.param == "shift5":
            bufs.append(n)                                         # j0, one byte per weight
        if w.calib == "batches":                                   # bf16 X, X^T, Y; accumulators
            et = w.experts * w.tokens
            bufs += ([2 * et * w.cols] if gram else
                     [2 * et * w.cols, 2 * et * w.cols, 2 * et * w.rows])
            bufs += [4 * L * n, 4 * n // w.group]
        bufs += [n, 8 * 17]                                        # initial codes; diagnostics
        expect = sum(_align(b) + 256 for b in bufs)
        assert lib.gsq_workspace_size(d) == expect, w.name
    # the largest workload fits comfortably in one GB300's HBM
    big = WORKLOADS["moe64_kquant3"]
    d = lib.make_desc(experts=big.experts, rows=big.rows, cols=big.cols, grid=big.grid, group_size=16,
                      scale_mode=lib.GSQ_SCALE_KQUANT2, lr_scales=0.0)
    assert lib.gsq_workspace_size(d) < 100e9


@pytest.mark.parametrize("sym", ["1", "0"])
def test_token_route_follows_the_flop_rule(lib, sym, monkeypatch):
    """A per-step-token layer on the tensor cores contracts through each micro-batch's
    Gram matrix exactly where that costs fewer flops than Y = D X^T, G = 2 Y X:
    C (T + 2R) < 4 R T with X^T X formed from its upper triangle, C (T + R) < 2 R T with
    every tile.  The route shows in the workspace (X^T and H against X, X^T and Y)."""
    monkeypatch.setenv("GSQ_TOKEN_SYM", sym)
    rule = ((lambda R, C, T: C * (T + 2 * R) < 4 * R * T) if sym == "1"
            else (lambda R, C, T: C * (T + R) < 2 * R * T))
    shapes = [(4096, 4096, 32768), (2048, 4096, 32768), (1024, 4096, 32768), (512, 4096, 32768),
              (4096, 4096, 2048), (4096, 1024, 8192), (136, 384, 328), (600, 384, 328)]
    picked = set()
    for R, C, T in shapes:
        d = lib.make_desc(experts=1, rows=R, cols=C, grid=(-1.5, -0.5, 0.5, 1.5), group_size=128,
                          calib_kind=lib.GSQ_CALIB_BATCHES, n_tokens=T)
        sizes = {}
        for route in ("gram", "direct"):
            monkeypatch.setenv("GSQ_TOKEN_ROUTE", route)
            sizes[route] = lib.gsq_workspace_size(d)
        monkeypatch.delenv("GSQ_TOKEN_ROUTE")
        assert sizes["gram"] != sizes["direct"], (R, C, T)
        want = "gram" if rule(R, C, T) else "direct"
        picked.add(want)
        assert lib.gsq_workspace_size(d) == sizes[want], (R, C, T, want)
    assert picked == {"gram", "direct"}


@pytest.mark.parametrize("kw,status", [
    (dict(cols=260), 2),                         # C % 8
    (dict(cols=192, group_size=128), 2),         # C % G
    (dict(group_size=96), 2),                    # not a power of two
    (dict(group_size=256), 2),
    (dict(grid=(0.5, -0.5)), 1),                 # not ascending
    (dict(grid=(1.0,)), 1),                      # K < 2
    (dict(grid=tuple(range(9))), 1),             # K > 8
    (dict(grid=(0.0, 0.0 + 1e-30)), 1),          # no level of usable magnitude? ascending but tiny ok
    (dict(rows=0), 2),
    (dict(cols=0), 2),                           # empty layers
    (dict(experts=0), 2),
    (dict(scale_mode=1, group_size=16), 1),      # KQUANT2 needs frozen scales
    (dict(scale_mode=1, group_size=16, lr_scales=0.0, cols=128), 2),   # C % 256
    (dict(w_dtype=7), 1),
    (dict(calib_kind=1, n_tokens=0), 1),
    (dict(gemm=5), 1),
    (dict(beta1=1.5), 1),
    (dict(calib_kind=2, n_tokens=0), 1),         # per-step batches need a token bound
    (dict(calib_kind=2, n_tokens=12), 1),        # ... that is a multiple of 8
    (dict(calib_kind=3), 1),
    (dict(param_mode=3), 1),                     # unknown parameterisation
    (dict(index_offset=4), 1),                   # a shard's noise offset is a multiple of 8
    (dict(index_offset=1 << 62), 1),             # ... and leaves room for the layer's indices
    (dict(param_mode=2), 1),                     # mask x sign needs {-a, 0, a}
    (dict(param_mode=2, grid=(-1.0, 0.0, 2.0)), 1),
    (dict(param_mode=2, grid=(-1.0, 0.5, 1.0)), 1),
])
def test_descriptor_validation(lib, kw, status):
    d = _desc(lib, **kw)
    if kw.get("grid") == (0.0, 1e-30):
        # ascending, finite, nonzero max level: valid
        assert lib.gsq_workspace_size(d) > 0
        return
    with pytest.raises(lib.GsqError) as ei:
        lib.gsq_workspace_size(d)
    assert ei.value.status == status
    assert lib.gsq_last_error()


def test_flags_known_and_unknown(lib):
    """Every documented flag bit is accepted (the unstaged-backward bit among them);
    a reserved or unknown bit is an argument error."""
    for f in (lib.GSQ_FLAG_NO_NOISE, lib.GSQ_FLAG_UNSTAGED,
              lib.GSQ_FLAG_NO_NOISE | lib.GSQ_FLAG_UNSTAGED):
        d = _desc(lib)
        d.flags = f
        assert lib.gsq_workspace_size(d) > 0
    for f in (2, 4, 16):
        d = _desc(lib)
        d.flags = f
        with pytest.raises(lib.GsqError) as ei:
            lib.gsq_workspace_size(d)
        assert ei.value.status == 1 and "flags" in lib.gsq_last_error()


def test_shard_offsets_accepted(lib):
    """A row shard (offset r0 * C) and an expert shard (offset e0 * R * C) are valid
    descriptors of the same size as the whole layer's piece."""
    base = lib.gsq_workspace_size(_desc(lib))
    assert lib.gsq_workspace_size(_desc(lib, index_offset=64 * 256)) == base
    assert lib.gsq_workspace_size(_desc(lib, index_offset=7 * 64 * 256)) == base


def test_parameterisations_size_their_logit_planes(lib):
    """The logit tensors hold K, 5 (local shift) or 2 (mask x sign) planes."""
    base = lib.gsq_workspace_size(_desc(lib, grid=(-1.0, 0.0, 1.0)))
    ms = lib.gsq_workspace_size(_desc(lib, grid=(-1.0, 0.0, 1.0), param_mode=2))
    sh = lib.gsq_workspace_size(_desc(lib, grid=(-1.0, 0.0, 1.0), param_mode=1))
    n = 64 * 256
    assert base - ms == 2 * 4 * n            # logits + momenta, one plane fewer
    assert sh - base == 2 * 2 * 4 * n + n + 256   # two planes more, plus j0 and its canary


def test_init_rejects_bad_buffers_before_cuda(lib):
    d = _desc(lib)
    nbytes = lib.gsq_workspace_size(d)
    with pytest.raises(lib.GsqError) as ei:      # W / calib missing
        lib.gsq_init_layer(d, 256, nbytes, 0)
    assert ei.value.status == lib.GSQ_ERR_INVALID_ARG
    d.W, d.calib = 4096, 8192
    with pytest.raises(lib.GsqError) as ei:      # workspace NULL
        lib.gsq_init_layer(d, 0, nbytes, 0)
    assert ei.value.status == lib.GSQ_ERR_WORKSPACE
    with pytest.raises(lib.GsqError) as ei:      # misaligned
        lib.gsq_init_layer(d, 256 + 16, nbytes, 0)
    assert ei.value.status == lib.GSQ_ERR_WORKSPACE
    with pytest.raises(lib.GsqError) as ei:      # too small
        lib.gsq_init_layer(d, 256, nbytes - 1, 0)
    assert ei.value.status == lib.GSQ_ERR_WORKSPACE and "too small" in lib.gsq_last_error()


def test_handle_checks(lib):
    for fn, args in [(lib._lib.gsq_step, (None, 0, 1.0, 1.0, 0.0, 1.0, None, None, None, None)),
                     (lib._lib.gsq_step, (12345678, 0, 1.0, 1.0, 0.0, 1.0, None, None, None, None)),
                     (lib._lib.gsq_project, (None, None, None, None)),
                     (lib._lib.gsq_destroy, (None,)),
                     (lib._lib.gsq_destroy, (987654321,)),
                     (lib._lib.gsq_sync_status, (None, None)),
                     (lib._lib.gsq_init_logits, (None, 4096, None, 1.0, 1.0, None)),
                     (lib._lib.gsq_init_logits, (24681357, 4096, None, 1.0, 1.0, None)),
                     (lib._lib.gsq_diagnose, (None, 1.0, 1.0, None, None))]:
        assert fn(*args) == lib.GSQ_ERR_INVALID_ARG
    assert lib.gsq_version().count(".") == 2


def test_fault_injection_env(tmp_path):
    code = textwrap.dedent(f"""
        import sys; sys.path.insert(0, {ROOT!r})
        from paper_2604_18556_gb300 import gsq
        d = gsq.make_desc(experts=1, rows=8, cols=128, grid=(-1.0, 0.0, 1.0), group_size=128)
        out = []
        for i in range(4):
            try:
                gsq.gsq_workspace_size(d); out.append(0)
            except gsq.GsqError as e:
                out.append(e.status)
        print(out)
    """)
    env = dict(os.environ, GSQ_FAULT_INJECT="gsq_workspace_size:3")
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env, check=True)
    assert r.stdout.strip() == "[0, 0, 8, 0]"
    env["GSQ_FAULT_INJECT"] = "gsq_init_layer:1"
    code2 = code.replace("gsq.gsq_workspace_size(d)", "gsq.gsq_init_layer(d, 256, 1 << 30, 0)")
    r = subprocess.run([sys.executable, "-c", code2], capture_output=True, text=True, env=env, check=True)
    assert r.stdout.strip() == "[8, 1, 1, 1]"   # injected first, then argument errors


def _noalloc_args(lib, **kw):
    a = lib.gsq_backward_args()
    a.num_experts, a.out_features, a.in_features = 1, 64, 256
    a.num_levels, a.group_size = 4, 128
    for k, q in enumerate((-1.5, -0.5, 0.5, 1.5)):
        a.grid[k] = q
    a.w_dtype, a.d_dtype = lib.GSQ_DTYPE_BF16, lib.GSQ_DTYPE_BF16
    # non-null stand-ins: every case below is rejected before any pointer is used
    a.W = a.G = a.logits = a.m_logits = a.scales = a.m_scales = 4096
    a.step, a.tau, a.kappa = 0, 1.0, 1.0
    for k, v in kw.items():
        if k == "grid":
            for i, q in enumerate(v):
                a.grid[i] = q
        else:
            setattr(a, k, v)
    return a


@pytest.mark.parametrize("kw,status,text", [
    (dict(in_features=260), 2, "C % 8"),
    (dict(in_features=0), 2, "C >= 8"),
    (dict(num_experts=0), 2, "E >= 1"),
    (dict(out_features=0), 2, "R >= 1"),
    (dict(num_levels=1), 1, "num_levels"),
    (dict(num_levels=9), 1, "num_levels"),
    (dict(group_size=96), 2, "group_size"),
    (dict(group_size=2), 2, "group_size"),
    (dict(group_size=256, in_features=512), 2, "group_size"),
    (dict(in_features=192), 2, "group_size"),            # C % G
    (dict(W=None), 1, "required"),
    (dict(G=None), 1, "required"),
    (dict(m_scales=None), 1, "required"),
    (dict(w_dtype=3), 1, "w_dtype"),
    (dict(d_dtype=-1), 1, "d_dtype"),
    (dict(flags=2), 1, "flags"),
    (dict(flags=8), 1, "flags"),
    (dict(step=1 << 32), 1, "step"),
    (dict(tau=0.0), 1, "tau"),
    (dict(tau=-1.0), 1, "tau"),
    (dict(tau=float("inf")), 1, "tau"),
    (dict(kappa=float("nan")), 1, "kappa"),
    (dict(grid=(-1.5, -0.5, -0.5, 1.5)), 1, "ascend"),
    (dict(out_features=4097, in_features=4096), 2, "16777216"),
])
def test_noalloc_validation_before_cuda(lib, kw, status, text):
    """gsq_backward_update_noalloc rejects every invalid argument on the host, before
    any CUDA call, with its status and a message naming the argument."""
    with pytest.raises(lib.GsqError) as ei:
        lib.gsq_backward_update_noalloc(_noalloc_args(lib, **kw), 0)
    assert ei.value.status == status
    assert text in lib.gsq_last_error(), lib.gsq_last_error()
    assert lib._lib.gsq_backward_update_noalloc(None, None) == lib.GSQ_ERR_INVALID_ARG
    assert "NULL" in lib.gsq_last_error()
