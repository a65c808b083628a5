"""The C ABI library without a GPU: it loads, exports every declared symbol, and rejects
bad arguments synchronously (before any CUDA call)."""
import ctypes
import os
import re
import subprocess

import pytest

from paper_2608_20172_gb300 import binding
from paper_2608_20172_gb300 import build as libbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "relation.h")


@pytest.fixture(scope="module")
def lib():
    libbuild.build()
    return binding.load()


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?\w+\s*\*?\s*(relation_\w+)\s*\(", src, re.M)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for n in ("relation_fwd", "relation_bwd", "relation_bwd_workspace_size",
              "relation_status_string"):
        assert n in names
    assert set(names) == set(binding.EXPORTED)


def test_library_exports_every_declared_symbol(lib):
    out = subprocess.run(["nm", "-D", "--defined-only", libbuild.LIB], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r"\s[TW]\s+(\w+)$", out, re.M))
    for n in declared_functions():
        assert n in exported, n
        assert getattr(lib, n) is not None


def test_status_strings(lib):
    for code, name in enumerate(["RELATION_OK", "RELATION_ERR_INVALID_ARG",
                                 "RELATION_ERR_UNSUPPORTED", "RELATION_ERR_ALIGNMENT",
                                 "RELATION_ERR_WORKSPACE", "RELATION_ERR_CUDA",
                                 "RELATION_ERR_TIMEOUT"]):
        assert binding.status_string(code) == name
    assert binding.status_string(99) == "RELATION_ERR_UNKNOWN"
    assert lib.relation_version() >> 16 == 1


def _shape(B=1, T=8, H=2, d=64, sB=None, sT=None, sH=None):
    sH = d if sH is None else sH
    sT = H * d if sT is None else sT
    sB = T * H * d if sB is None else sB
    return binding.Shape(B, T, H, d, sB, sT, sH)


def _fwd(lib, ptrs, shape, dt=binding.BF16, lam=0.5, tau=2.0, kernel=0):
    q, k, v, o, lz = ptrs
    return lib.relation_fwd_ex(q, k, v, o, lz, lam, tau, shape, dt, kernel, None, None)


GOOD = [0x10000, 0x20000, 0x30000, 0x40000, 0x50000]  # aligned, never dereferenced here


@pytest.mark.parametrize("case,expect", [
    ("null q", binding.ERR_INVALID_ARG),
    ("misaligned v", binding.ERR_ALIGNMENT),
    ("T = 0", binding.ERR_INVALID_ARG),
    ("d = 36", binding.ERR_UNSUPPORTED),
    ("d = 136", binding.ERR_UNSUPPORTED),
    ("odd stride", binding.ERR_ALIGNMENT),
    ("tau = 0", binding.ERR_INVALID_ARG),
    ("lambda inf", binding.ERR_INVALID_ARG),
    ("bad dtype", binding.ERR_INVALID_ARG),
    ("tcgen05 for fp32", binding.ERR_UNSUPPORTED),
    ("too many heads", binding.ERR_UNSUPPORTED),
])
def test_fwd_rejects_bad_arguments(lib, case, expect):
    ptrs, shape, kw = list(GOOD), _shape(), {}
    if case == "null q":
        ptrs[0] = None
    elif case == "misaligned v":
        ptrs[2] = 0x30008
    elif case == "T = 0":
        shape = _shape(T=0)
    elif case == "d = 36":
        shape = _shape(d=36)
    elif case == "d = 136":
        shape = _shape(d=136)
    elif case == "odd stride":
        shape = _shape(sT=130)
    elif case == "tau = 0":
        kw["tau"] = 0.0
    elif case == "lambda inf":
        kw["lam"] = float("inf")
    elif case == "bad dtype":
        kw["dt"] = 7
    elif case == "tcgen05 for fp32":
        kw["dt"], kw["kernel"] = binding.F32, 2
    elif case == "too many heads":
        shape = _shape(B=300, H=300)
    assert _fwd(lib, ptrs, shape, **kw) == expect


def test_bwd_workspace_rules(lib):
    shape = _shape(B=2, T=100, H=3, d=64)
    need = lib.relation_bwd_workspace_size(shape, binding.BF16)
    rows = 2 * 3 * 100
    assert need >= rows * 64 * 4 + 3 * rows * 4
    assert lib.relation_bwd_workspace_size(_shape(T=0), binding.BF16) == 0
    p = [ctypes.c_void_p(0x10000 * (i + 1)) for i in range(10)]
    args = p[:9] + [p[9]]
    rc = lib.relation_bwd_ex(*args, 0.5, 2.0, shape, binding.BF16, ctypes.c_void_p(0x100000),
                             need - 1, 0, None, None)
    assert rc == binding.ERR_WORKSPACE
    rc = lib.relation_bwd_ex(*args, 0.5, 2.0, shape, binding.BF16, None, need, 0, None, None)
    assert rc == binding.ERR_WORKSPACE
    rc = lib.relation_bwd_ex(*args, 0.5, 2.0, shape, binding.BF16, ctypes.c_void_p(0x100010),
                             need, 0, None, None)
    assert rc == binding.ERR_ALIGNMENT
    rc = lib.relation_bwd_ex(*p[:9], None, 0.5, 2.0, shape, binding.BF16,
                             ctypes.c_void_p(0x100000), need, 0, None, None)
    assert rc == binding.ERR_INVALID_ARG


def test_selftest_argument_checks(lib):
    assert lib.relation_selftest_wait_timeout(None, 10, None) == binding.ERR_INVALID_ARG
    assert lib.relation_selftest_wait_timeout(ctypes.c_void_p(0x1000), 0, None) == \
        binding.ERR_INVALID_ARG
    assert lib.relation_selftest_wait_timeout(ctypes.c_void_p(0x1002), 10, None) == \
        binding.ERR_ALIGNMENT


def test_binding_refuses_cpu_tensors():
    import torch
    x = torch.zeros(1, 4, 1, 64, dtype=torch.bfloat16)
    with pytest.raises(ValueError):
        binding.fwd(x, x, x, 0.5)


def test_missing_library_fails_loudly(tmp_path):
    with pytest.raises(binding.RelationLibraryMissing):
        binding.load(str(tmp_path / "nope.so"))


@pytest.mark.parametrize("case,expect", [
    ("odd H", binding.ERR_UNSUPPORTED),
    ("d = 36", binding.ERR_UNSUPPORTED),
    ("d = 264", binding.ERR_UNSUPPORTED),
    ("pairing 2", binding.ERR_INVALID_ARG),
    ("base 0", binding.ERR_INVALID_ARG),
    ("null theta", binding.ERR_INVALID_ARG),
    ("misaligned k", binding.ERR_ALIGNMENT),
    ("odd stride", binding.ERR_ALIGNMENT),
])
def test_layer_prep_rejects_bad_arguments(lib, case, expect):
    p = [ctypes.c_void_p(0x10000 * (i + 1)) for i in range(6)]
    theta = ctypes.c_void_p(0x90000)
    shape, pairing, base = _shape(H=4), 0, 1.0e4
    if case == "odd H":
        shape = _shape(H=3)
    elif case == "d = 36":
        shape = _shape(H=4, d=36)
    elif case == "d = 264":
        shape = _shape(H=4, d=264)
    elif case == "pairing 2":
        pairing = 2
    elif case == "base 0":
        base = 0.0
    elif case == "null theta":
        theta = None
    elif case == "misaligned k":
        p[4] = ctypes.c_void_p(0x50008)
    elif case == "odd stride":
        shape = _shape(H=4, sT=260)
    rc = lib.relation_layer_prep(p[0], p[1], p[2], theta, pairing, base, p[3], p[4], p[5], shape,
                                 binding.BF16, None)
    assert rc == expect


def test_layer_grad_workspace_rules(lib):
    shape = _shape(B=2, T=100, H=4, d=64)
    need = lib.relation_layer_grad_workspace_size(shape, binding.BF16)
    assert need == 2 * ((100 + 15) // 16) * 2 * 4  # one fp32 partial per CTA and head pair
    assert lib.relation_layer_grad_workspace_size(_shape(H=3), binding.BF16) == 0
    p = [ctypes.c_void_p(0x10000 * (i + 1)) for i in range(7)]
    theta, dtheta = ctypes.c_void_p(0x90000), ctypes.c_void_p(0xA0000)
    rc = lib.relation_layer_grad(p[0], p[1], p[2], p[3], theta, 0, 1.0e4, p[4], p[5], p[6], dtheta,
                                 shape, binding.BF16, ctypes.c_void_p(0x100000), need - 1, None)
    assert rc == binding.ERR_WORKSPACE
    rc = lib.relation_layer_grad(p[0], p[1], p[2], p[3], theta, 0, 1.0e4, p[4], p[5], p[6], None,
                                 shape, binding.BF16, ctypes.c_void_p(0x100000), need, None)
    assert rc == binding.ERR_INVALID_ARG


@pytest.mark.parametrize("case,expect", [
    ("d = 48", binding.ERR_UNSUPPORTED),
    ("stride not a multiple of 4", binding.ERR_ALIGNMENT),
    ("null alpha", binding.ERR_INVALID_ARG),
    ("tau = 0", binding.ERR_INVALID_ARG),
    ("misaligned y", binding.ERR_ALIGNMENT),
])
def test_linear_rejects_bad_arguments(lib, case, expect):
    p = [ctypes.c_void_p(0x10000 * (i + 1)) for i in range(5)]
    shape, tau = _shape(d=64), 2.0
    if case == "d = 48":
        shape = _shape(d=48)
    elif case == "stride not a multiple of 4":
        shape = _shape(d=64, sH=66, sT=2 * 66, sB=8 * 2 * 66)
    elif case == "null alpha":
        p[3] = None
    elif case == "tau = 0":
        tau = 0.0
    elif case == "misaligned y":
        p[4] = ctypes.c_void_p(0x50004)
    rc = lib.relation_linear_fwd(p[0], p[1], p[2], p[3], p[4], tau, shape, binding.BF16, None,
                                 None)
    assert rc == expect


@pytest.mark.parametrize("case,expect", [
    ("tcgen05 fp32", binding.ERR_UNSUPPORTED),
    ("tcgen05 d = 32", binding.ERR_UNSUPPORTED),
    ("tcgen05 stride not a multiple of 8", binding.ERR_ALIGNMENT),
    ("unknown family", binding.ERR_INVALID_ARG),
])
def test_linear_fwd_ex_family_rules(lib, case, expect):
    """The chunked tensor-core family serves bf16 with d_h 64 or 128 and element strides
    that are multiples of 8; other requests for it are refused with nothing launched."""
    p = [ctypes.c_void_p(0x10000 * (i + 1)) for i in range(5)]
    shape, dt, fam = _shape(d=64), binding.BF16, binding.KERNELS["tcgen05"]
    if case == "tcgen05 fp32":
        dt = binding.F32
    elif case == "tcgen05 d = 32":
        shape = _shape(d=32)
    elif case == "tcgen05 stride not a multiple of 8":
        shape = _shape(d=64, sH=68, sT=2 * 68, sB=8 * 2 * 68)
    elif case == "unknown family":
        fam = 7
    rc = lib.relation_linear_fwd_ex(p[0], p[1], p[2], p[3], p[4], 2.0, shape, dt, fam, None, None)
    assert rc == expect


def test_linear_fwd_ws_workspace_rules(lib):
    """The chunk-parallel forward's workspace: B H (d/64) ceil(T/128) d rows of 64 fp32 dC and
    one fp32 decay, B H (d/64) (ceil(T/128) + 1) d rows of 64 bf16 states, each array padded
    to 256 bytes; fp32 and
    other widths need none; a short or misaligned workspace is refused before any launch."""
    shape = _shape(B=1, T=300, H=2, d=64)
    rows, rows_c0 = 1 * 2 * 1 * 3 * 64, 1 * 2 * 1 * 4 * 64  # C0: every block's and the final
    pad = lambda x: (x + 255) // 256 * 256
    need = lib.relation_linear_fwd_workspace_size(shape, binding.BF16)
    assert need == pad(rows * 64 * 4) + pad(rows * 4) + pad(rows_c0 * 64 * 2)
    assert lib.relation_linear_fwd_workspace_size(shape, binding.F32) == 0
    assert lib.relation_linear_fwd_workspace_size(_shape(d=32), binding.BF16) == 0
    p = [ctypes.c_void_p(0x10000 * (i + 1)) for i in range(5)]
    rc = lib.relation_linear_fwd_ws(*p, 2.0, shape, binding.BF16, ctypes.c_void_p(0x100000),
                                    need - 1, None, None)
    assert rc == binding.ERR_WORKSPACE
    rc = lib.relation_linear_fwd_ws(*p, 2.0, shape, binding.BF16, ctypes.c_void_p(0x100008),
                                    need, None, None)
    assert rc == binding.ERR_ALIGNMENT


def test_linear_bwd_workspace_rules(lib):
    shape = _shape(B=2, T=20, H=3, d=64)
    simt = lib.relation_linear_bwd_ex_workspace_size(shape, binding.BF16, binding.KERNELS["simt"])
    # checkpoints every 8 tokens (3 of 64 x 64) plus the column splits' partial row sums
    assert simt == (2 * 3 * 3 * 64 * 64 + 2 * 3 * 2 * 20 * 3 * 64) * 4
    # the chunked family, one 128-token block per head (6 heads): fp32 rows of 64 and the
    # decays, the states entering the block and the final one, the adjoints (bf16)
    tc = lib.relation_linear_bwd_ex_workspace_size(shape, binding.BF16, binding.KERNELS["tcgen05"])
    assert tc == 6 * 64 * 64 * 4 + 6 * 64 * 4 + 6 * 2 * 64 * 64 * 2 + 6 * 64 * 64 * 2
    need = lib.relation_linear_bwd_workspace_size(shape, binding.BF16)
    assert need == tc  # AUTO takes the chunked kernel for bf16 at d_h = 64
    assert lib.relation_linear_bwd_ex_workspace_size(shape, binding.F32,
                                                     binding.KERNELS["tcgen05"]) == 0
    assert lib.relation_linear_bwd_workspace_size(shape, binding.F32) == simt
    d128 = _shape(B=2, T=20, H=3, d=128)
    assert lib.relation_linear_bwd_ex_workspace_size(d128, binding.BF16,
                                                     binding.KERNELS["tcgen05"]) == 0
    assert lib.relation_linear_bwd_workspace_size(d128, binding.BF16) == \
        lib.relation_linear_bwd_ex_workspace_size(d128, binding.BF16, binding.KERNELS["simt"])
    assert lib.relation_linear_bwd_workspace_size(_shape(d=48), binding.BF16) == 0
    p = [ctypes.c_void_p(0x10000 * (i + 1)) for i in range(9)]
    rc = lib.relation_linear_bwd(*p, 2.0, shape, binding.BF16, ctypes.c_void_p(0x100000), need - 1,
                                 None, None)
    assert rc == binding.ERR_WORKSPACE
    rc = lib.relation_linear_bwd_ex(*p, 2.0, shape, binding.BF16, binding.KERNELS["simt"],
                                    ctypes.c_void_p(0x100000), simt - 1, None, None)
    assert rc == binding.ERR_WORKSPACE
    rc = lib.relation_linear_bwd_ex(*p, 2.0, shape, binding.BF16, binding.KERNELS["tcgen05"],
                                    ctypes.c_void_p(0x100008), tc, None, None)
    assert rc == binding.ERR_ALIGNMENT
    rc = lib.relation_linear_bwd_ex(*p, 2.0, shape, binding.F32, binding.KERNELS["tcgen05"],
                                    ctypes.c_void_p(0x100000), 1 << 30, None, None)
    assert rc == binding.ERR_UNSUPPORTED
    odd = _shape(B=2, T=20, H=3, d=64)
    odd.sB, odd.sT, odd.sH = 20 * 3 * 68, 3 * 68, 68
    rc = lib.relation_linear_bwd_ex(*p, 2.0, odd, binding.BF16, binding.KERNELS["tcgen05"],
                                    ctypes.c_void_p(0x100000), 1 << 30, None, None)
    assert rc == binding.ERR_ALIGNMENT
    rc = lib.relation_linear_bwd_ex(*p, 2.0, shape, binding.BF16, 7, ctypes.c_void_p(0x100000),
                                    1 << 30, None, None)
    assert rc == binding.ERR_INVALID_ARG


@pytest.mark.parametrize("case,expect", [
    ("d = 136", binding.ERR_UNSUPPORTED),
    ("null lengths", binding.ERR_INVALID_ARG),
    ("lambda nan", binding.ERR_INVALID_ARG),
    ("small workspace", binding.ERR_WORKSPACE),
    ("q stride 0", binding.ERR_INVALID_ARG),
])
def test_decode_rejects_bad_arguments(lib, case, expect):
    p = [ctypes.c_void_p(0x10000 * (i + 1)) for i in range(6)]
    cache, lam, qsB, qsH = _shape(B=2, T=64, H=2, d=64), 0.5, 128, 64
    need = lib.relation_decode_workspace_size(cache, binding.BF16)
    ws = need
    if case == "d = 136":
        cache = _shape(B=2, T=64, H=2, d=136)
    elif case == "null lengths":
        p[3] = None
    elif case == "lambda nan":
        lam = float("nan")
    elif case == "small workspace":
        ws = need - 1
    elif case == "q stride 0":
        qsB = 0
    rc = lib.relation_decode(p[0], p[1], p[2], p[3], p[4], p[5], lam, 2.0, cache, qsB, qsH,
                             binding.BF16, ctypes.c_void_p(0x100000), ws, None, None)
    assert rc == expect


def test_context_parallel_entry_points_reject_bad_arguments(lib):
    """The context-parallel calls check their arguments on the host and launch nothing."""
    q = _shape(B=2, T=100, H=3, d=64)
    kv = _shape(B=2, T=40, H=3, d=64)
    p = [ctypes.c_void_p(0x10000 * (i + 1)) for i in range(6)]
    st = lambda *a: lib.relation_fwd_state(*p, *a, None, None)
    assert st(q, kv, 0, binding.F32) == binding.ERR_UNSUPPORTED  # tensor-core tiles: bf16
    assert st(q, kv, 2, binding.BF16) == binding.ERR_INVALID_ARG
    assert st(q, kv, 1, binding.BF16) == binding.ERR_INVALID_ARG  # causal: T_k = T_q
    assert st(q, _shape(B=2, T=40, H=4, d=64), 0, binding.BF16) == binding.ERR_INVALID_ARG
    assert st(_shape(B=2, T=100, H=3, d=136), _shape(B=2, T=40, H=3, d=136), 0,
              binding.BF16) == binding.ERR_UNSUPPORTED
    assert lib.relation_fwd_state(*p[:3], None, *p[4:], q, kv, 0, binding.BF16, None,
                                  None) == binding.ERR_INVALID_ARG
    assert lib.relation_fwd_state(*p[:3], ctypes.c_void_p(0x10004), *p[4:], q, kv, 0,
                                  binding.BF16, None, None) == binding.ERR_ALIGNMENT
    assert lib.relation_state_merge(*p, _shape(d=132), None) == binding.ERR_UNSUPPORTED
    assert lib.relation_state_merge(*p, _shape(T=0), None) == binding.ERR_INVALID_ARG
    f = [ctypes.c_void_p(0x10000 * (i + 1)) for i in range(8)]
    fin = lambda pos0, shp=q, lam=0.5: lib.relation_state_finish(*f, None, lam, 2.0, pos0, shp,
                                                                 binding.BF16, None)
    assert fin(-1) == binding.ERR_INVALID_ARG
    assert fin(0, lam=float("nan")) == binding.ERR_INVALID_ARG
    assert fin(0, shp=_shape(d=136)) == binding.ERR_UNSUPPORTED
