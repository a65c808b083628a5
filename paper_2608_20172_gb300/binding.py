"""Thin ctypes binding of librelation (include/relation.h) for torch CUDA tensors.

Argument marshalling only: every step of the operator runs in the library's CUDA
kernels.  Tensors are [B, T, H, d_h] (any strides with d_h contiguous, the same for
all tensors of a call); logZ is a dense fp32 [B, H, T].  Calls are enqueued on the
current torch CUDA stream unless ``stream`` is given.

Loading fails loudly (``RelationLibraryMissing``) when the compiled library is absent:
there is no CPU fallback.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "librelation.so")

# relation_status
OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_ALIGNMENT, ERR_WORKSPACE, ERR_CUDA, ERR_TIMEOUT = range(7)
# relation_dtype
F32, BF16 = 0, 1
# relation_kernel
KERNELS = {"auto": 0, "simt": 1, "tcgen05": 2}

EXPORTED = ("relation_fwd", "relation_fwd_ex", "relation_bwd", "relation_bwd_ex",
            "relation_bwd_workspace_size", "relation_status_string", "relation_version",
            "relation_selftest_wait_timeout", "relation_launch_count", "relation_last_cuda_error",
            "relation_bwd_stages", "relation_bwd_static", "relation_fwd_flow",
            "relation_decode", "relation_decode_workspace_size", "relation_fwd_state",
            "relation_state_merge", "relation_state_finish", "relation_linear_fwd",
            "relation_linear_fwd_ex", "relation_linear_fwd_ws",
            "relation_linear_fwd_workspace_size",
            "relation_linear_bwd", "relation_linear_bwd_workspace_size",
            "relation_linear_bwd_ex", "relation_linear_bwd_ex_workspace_size", "relation_layer_prep",
            "relation_layer_grad", "relation_layer_grad_workspace_size")


class RelationLibraryMissing(RuntimeError):
    pass


class RelationError(RuntimeError):
    def __init__(self, code: int, where: str):
        msg = f"{where}: {status_string(code)} ({code})"
        if code == ERR_CUDA:
            msg += f": {load().relation_last_cuda_error().decode()}"
        super().__init__(msg)
        self.code = code


class Shape(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int), ("T", ctypes.c_int), ("H", ctypes.c_int),
                ("d_h", ctypes.c_int), ("sB", ctypes.c_longlong), ("sT", ctypes.c_longlong),
                ("sH", ctypes.c_longlong)]


_lock = threading.Lock()
_lib = None


def load(path: str | None = None):
    """Load librelation.so (default: the in-tree build) and declare its signatures."""
    global _lib
    with _lock:
        if _lib is not None and path is None:
            return _lib
        p = path or LIB_PATH
        if not os.path.exists(p):
            raise RelationLibraryMissing(
                f"{p} not found: build it with paper_2608_20172_gb300.build.build()")
        lib = ctypes.CDLL(p)
        vp, ip = ctypes.c_void_p, ctypes.c_void_p
        f, i, sz = ctypes.c_float, ctypes.c_int, ctypes.c_size_t
        lib.relation_fwd.argtypes = [vp, vp, vp, vp, vp, f, f, Shape, i, ip, vp]
        lib.relation_fwd_ex.argtypes = [vp, vp, vp, vp, vp, f, f, Shape, i, i, ip, vp]
        lib.relation_fwd_flow.argtypes = [vp, vp, vp, vp, vp, vp, f, f, Shape, i, i, ip, vp]
        ll = ctypes.c_longlong
        lib.relation_decode.argtypes = [vp, vp, vp, vp, vp, vp, f, f, Shape, ll, ll, i, vp,
                                        ctypes.c_size_t, ip, vp]
        lib.relation_decode_workspace_size.argtypes = [Shape, i]
        lib.relation_fwd_state.argtypes = [vp, vp, vp, vp, vp, vp, Shape, Shape, i, i, ip, vp]
        lib.relation_state_merge.argtypes = [vp, vp, vp, vp, vp, vp, Shape, vp]
        lib.relation_state_finish.argtypes = [vp, vp, vp, vp, vp, vp, vp, vp, vp, f, f, ll, Shape,
                                              i, vp]
        lib.relation_linear_fwd.argtypes = [vp, vp, vp, vp, vp, f, Shape, i, ip, vp]
        lib.relation_linear_fwd_ex.argtypes = [vp, vp, vp, vp, vp, f, Shape, i, i, ip, vp]
        lib.relation_linear_fwd_ws.argtypes = [vp, vp, vp, vp, vp, f, Shape, i, vp, sz, ip, vp]
        lib.relation_linear_fwd_workspace_size.argtypes = [Shape, i]
        lib.relation_linear_fwd_workspace_size.restype = sz
        lib.relation_linear_bwd.argtypes = [vp, vp, vp, vp, vp, vp, vp, vp, vp, f, Shape, i, vp,
                                            ctypes.c_size_t, ip, vp]
        lib.relation_linear_bwd_workspace_size.argtypes = [Shape, i]
        lib.relation_linear_bwd_ex.argtypes = [vp, vp, vp, vp, vp, vp, vp, vp, vp, f, Shape, i, i,
                                               vp, sz, ip, vp]
        lib.relation_linear_bwd_ex_workspace_size.argtypes = [Shape, i, i]
        lib.relation_linear_bwd_ex_workspace_size.restype = sz
        lib.relation_layer_prep.argtypes = [vp, vp, vp, vp, i, f, vp, vp, vp, Shape, i, vp]
        lib.relation_layer_grad.argtypes = [vp, vp, vp, vp, vp, i, f, vp, vp, vp, vp, Shape, i,
                                            vp, sz, vp]
        lib.relation_layer_grad_workspace_size.argtypes = [Shape, i]
        lib.relation_layer_grad_workspace_size.restype = sz
        lib.relation_linear_bwd_workspace_size.restype = ctypes.c_size_t
        lib.relation_decode_workspace_size.restype = ctypes.c_size_t
        lib.relation_bwd.argtypes = [vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, f, f, Shape, i, vp,
                                     sz, ip, vp]
        lib.relation_bwd_ex.argtypes = [vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, f, f, Shape, i,
                                        vp, sz, i, ip, vp]
        lib.relation_bwd_stages.argtypes = [vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, f, f, Shape,
                                            i, vp, sz, i, ctypes.c_uint, ip, vp]
        lib.relation_bwd_stages.restype = ctypes.c_int
        lib.relation_bwd_static.argtypes = [vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, f, f, Shape,
                                            i, i, ip, vp]
        lib.relation_bwd_static.restype = ctypes.c_int
        lib.relation_bwd_workspace_size.argtypes = [Shape, i]
        lib.relation_bwd_workspace_size.restype = sz
        lib.relation_status_string.argtypes = [i]
        lib.relation_status_string.restype = ctypes.c_char_p
        lib.relation_version.argtypes = []
        lib.relation_selftest_wait_timeout.argtypes = [ip, i, vp]
        lib.relation_launch_count.argtypes = [i, i, i, i]
        lib.relation_last_cuda_error.argtypes = []
        lib.relation_last_cuda_error.restype = ctypes.c_char_p
        for n in ("relation_fwd", "relation_fwd_ex", "relation_bwd", "relation_bwd_ex",
                  "relation_version", "relation_selftest_wait_timeout", "relation_launch_count"):
            getattr(lib, n).restype = ctypes.c_int
        if path is None:
            _lib = lib
        return lib


def status_string(code: int) -> str:
    return load().relation_status_string(int(code)).decode()


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return F32
    if t.dtype == torch.bfloat16:
        return BF16
    raise TypeError(f"unsupported dtype {t.dtype}")


def shape_of(t: torch.Tensor) -> Shape:
    """relation_shape of a [B, T, H, d_h] tensor with d_h contiguous."""
    if t.dim() != 4:
        raise ValueError("expected a [B, T, H, d_h] tensor")
    if t.stride(3) != 1:
        raise ValueError("d_h must be contiguous")
    B, T, H, d = t.shape
    return Shape(B, T, H, d, t.stride(0), t.stride(1), t.stride(2))


def _same_layout(ref: torch.Tensor, *others: torch.Tensor):
    for o in others:
        if o.shape != ref.shape or o.stride() != ref.stride() or o.dtype != ref.dtype:
            raise ValueError("all tensors of a call need the same shape, strides and dtype")
        if not o.is_cuda or o.device != ref.device:
            raise ValueError("all tensors must live on the same CUDA device")


def _like(t: torch.Tensor) -> torch.Tensor:
    """An output with t's shape, dtype, device and strides.  The C ABI writes an output
    with its input's element strides, which torch.empty_like does not keep for a view that
    is not dense (e.g. a slice of a padded tensor)."""
    return torch.empty_strided(t.size(), t.stride(), dtype=t.dtype, device=t.device)


def _stream(stream) -> int:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def workspace_size(q: torch.Tensor) -> int:
    return int(load().relation_bwd_workspace_size(shape_of(q), _dtype_code(q)))


def fwd(q, k, v, lam: float, tau_s: float = 2.0, *, kernel: str = "auto", out=None, logz=None,
        dev_status=None, stream=None):
    """Forward.  Returns (Y, logZ)."""
    _same_layout(q, k, v)
    B, T, H, _ = q.shape
    if out is None:
        out = _like(q)
    _same_layout(q, out)
    if logz is None:
        logz = torch.empty((B, H, T), device=q.device, dtype=torch.float32)
    rc = load().relation_fwd_ex(_ptr(q), _ptr(k), _ptr(v), _ptr(out), _ptr(logz), float(lam),
                                float(tau_s), shape_of(q), _dtype_code(q), KERNELS[kernel],
                                _ptr(dev_status), ctypes.c_void_p(_stream(stream)))
    if rc != OK:
        raise RelationError(rc, "relation_fwd")
    return out, logz


def fwd_flow(q, k, v, lam: float, tau_s: float = 2.0, *, kernel: str = "auto", out=None,
             logz=None, self_flow=None, dev_status=None, stream=None):
    """Forward with the Self flow F_ii = 1 - g_i of every row as a side output.
    Returns (Y, logZ, F_self) with F_self [B, H, T] fp32."""
    _same_layout(q, k, v)
    B, T, H, _ = q.shape
    if out is None:
        out = _like(q)
    _same_layout(q, out)
    if logz is None:
        logz = torch.empty((B, H, T), device=q.device, dtype=torch.float32)
    if self_flow is None:
        self_flow = torch.empty((B, H, T), device=q.device, dtype=torch.float32)
    rc = load().relation_fwd_flow(_ptr(q), _ptr(k), _ptr(v), _ptr(out), _ptr(logz),
                                  _ptr(self_flow), float(lam), float(tau_s), shape_of(q),
                                  _dtype_code(q), KERNELS[kernel], _ptr(dev_status),
                                  ctypes.c_void_p(_stream(stream)))
    if rc != OK:
        raise RelationError(rc, "relation_fwd_flow")
    return out, logz, self_flow


def linear_fwd(p1, p2, v, alpha, tau_s: float = 2.0, *, kernel: str = "auto", out=None,
               dev_status=None, stream=None):
    """Linear Relation forward.  p1, p2, v [B, T, H, d] (fp32 or bf16), alpha [B, T, H, d]
    fp32 with p1's strides.  ``kernel``: "simt" (the recurrence), "tcgen05" (the chunked
    tensor-core form) or "auto".  Returns Y."""
    _same_layout(p1, p2, v)
    if alpha.dtype != torch.float32 or tuple(alpha.shape) != tuple(p1.shape) or \
            tuple(alpha.stride()) != tuple(p1.stride()):
        raise ValueError("alpha must be fp32 with p1's shape and strides")
    out = _like(p1) if out is None else out
    _same_layout(p1, out)
    rc = load().relation_linear_fwd_ex(_ptr(p1), _ptr(p2), _ptr(v), _ptr(alpha), _ptr(out),
                                       float(tau_s), shape_of(p1), _dtype_code(p1),
                                       KERNELS[kernel], _ptr(dev_status),
                                       ctypes.c_void_p(_stream(stream)))
    if rc != OK:
        raise RelationError(rc, "relation_linear_fwd_ex")
    return out


def _check_summary(state, B, H, T, d, device):
    """(m, l, z): dense fp32 [B, H, T], [B, H, T], [B, H, T, d] on `device`."""
    m, l, z = state
    for t, shp in ((m, (B, H, T)), (l, (B, H, T)), (z, (B, H, T, d))):
        if tuple(t.shape) != shp or t.dtype != torch.float32 or not t.is_contiguous() or \
                t.device != device:
            raise ValueError("an Exchange summary is dense fp32 (m, l [B, H, T], z [B, H, T, d]) "
                             "on the operands' device")


def fwd_state(q, k, v, causal: bool, *, out=None, dev_status=None, stream=None):
    """Exchange summary of every row of q ([B, Tq, H, d]) over the keys of k, v ([B, Tk, H,
    d]): causal = the queries' own tokens (keys before each row), else every key precedes
    every query.  Returns (m, l, z): m, l [B, H, Tq] and z [B, H, Tq, d], fp32."""
    _same_layout(k, v)
    if causal:
        _same_layout(q, k, v)
    B, Tq, H, d = q.shape
    if out is None:
        out = (torch.empty((B, H, Tq), dtype=torch.float32, device=q.device),
               torch.empty((B, H, Tq), dtype=torch.float32, device=q.device),
               torch.empty((B, H, Tq, d), dtype=torch.float32, device=q.device))
    m, l, z = out
    _check_summary(out, B, H, Tq, d, q.device)
    rc = load().relation_fwd_state(_ptr(q), _ptr(k), _ptr(v), _ptr(m), _ptr(l), _ptr(z),
                                   shape_of(q), shape_of(k), int(bool(causal)), _dtype_code(q),
                                   _ptr(dev_status), ctypes.c_void_p(_stream(stream)))
    if rc != OK:
        raise RelationError(rc, "relation_fwd_state")
    return m, l, z


def state_merge(state, other, *, stream=None):
    """Merge the summary ``other`` into ``state`` (both (m, l, z) as fwd_state returns them,
    same rows) in place; returns ``state``."""
    m, l, z = state
    m2, l2, z2 = other
    B, H, T, d = z.shape
    _check_summary(state, B, H, T, d, z.device)
    _check_summary(other, B, H, T, d, z.device)
    rc = load().relation_state_merge(_ptr(m), _ptr(l), _ptr(z), _ptr(m2), _ptr(l2), _ptr(z2),
                                     Shape(B, T, H, d, T * H * d, H * d, d),
                                     ctypes.c_void_p(_stream(stream)))
    if rc != OK:
        raise RelationError(rc, "relation_state_merge")
    return state


def state_finish(q, k, v, state, lam: float, tau_s: float = 2.0, pos0: int = 0, *, out=None,
                 logz=None, self_flow=None, stream=None):
    """Y and logZ of the rows of q, k, v from their merged summary ``state``; row r is at
    zero-based position pos0 + r of the sequence.  Returns (Y, logZ)."""
    _same_layout(q, k, v)
    m, l, z = state
    B, T, H, d = q.shape
    out = _like(q) if out is None else out
    _same_layout(q, out)
    logz = torch.empty((B, H, T), dtype=torch.float32, device=q.device) if logz is None else logz
    _check_summary(state, B, H, T, d, q.device)
    if tuple(logz.shape) != (B, H, T) or logz.dtype != torch.float32 or not logz.is_contiguous():
        raise ValueError("logz must be a dense fp32 [B, H, T] tensor")
    rc = load().relation_state_finish(_ptr(q), _ptr(k), _ptr(v), _ptr(m), _ptr(l), _ptr(z),
                                      _ptr(out), _ptr(logz), _ptr(self_flow), float(lam),
                                      float(tau_s), int(pos0), shape_of(q), _dtype_code(q),
                                      ctypes.c_void_p(_stream(stream)))
    if rc != OK:
        raise RelationError(rc, "relation_state_finish")
    return out, logz


def linear_fwd_workspace_size(p1) -> int:
    return int(load().relation_linear_fwd_workspace_size(shape_of(p1), _dtype_code(p1)))


def linear_fwd_ws(p1, p2, v, alpha, tau_s: float = 2.0, *, workspace=None, out=None,
                  dev_status=None, stream=None):
    """Linear Relation forward through relation_linear_fwd_ws (the chunk-parallel form for
    long sequences with few heads).  ``workspace``: a uint8 CUDA tensor of at least
    linear_fwd_workspace_size(p1) bytes (allocated here when None).  Returns Y."""
    _same_layout(p1, p2, v)
    if alpha.dtype != torch.float32 or tuple(alpha.shape) != tuple(p1.shape) or \
            tuple(alpha.stride()) != tuple(p1.stride()):
        raise ValueError("alpha must be fp32 with p1's shape and strides")
    out = _like(p1) if out is None else out
    _same_layout(p1, out)
    need = linear_fwd_workspace_size(p1)
    if workspace is None:
        workspace = torch.empty(max(need, 16), dtype=torch.uint8, device=p1.device)
    rc = load().relation_linear_fwd_ws(_ptr(p1), _ptr(p2), _ptr(v), _ptr(alpha), _ptr(out),
                                       float(tau_s), shape_of(p1), _dtype_code(p1),
                                       _ptr(workspace), workspace.numel(), _ptr(dev_status),
                                       ctypes.c_void_p(_stream(stream)))
    if rc != OK:
        raise RelationError(rc, "relation_linear_fwd_ws")
    return out


def linear_bwd_workspace_size(p1, kernel: str = "auto") -> int:
    """Bytes of device scratch linear_bwd needs for tensors shaped like p1 (0: the kernel
    family does not serve this request)."""
    return int(load().relation_linear_bwd_ex_workspace_size(shape_of(p1), _dtype_code(p1),
                                                            KERNELS[kernel]))


def linear_bwd(p1, p2, v, alpha, dy, tau_s: float = 2.0, *, kernel: str = "auto",
               workspace=None, dev_status=None, stream=None):
    """Linear Relation backward.  Returns (dp1, dp2, dv, dalpha) with dalpha fp32.
    ``kernel``: "auto", "simt" (reverse mode through the token recurrence) or "tcgen05"
    (through the 128-token blocks of the chunked forward; bf16, d_h 64)."""
    _same_layout(p1, p2, v, dy)
    if alpha.dtype != torch.float32 or tuple(alpha.shape) != tuple(p1.shape) or \
            tuple(alpha.stride()) != tuple(p1.stride()):
        raise ValueError("alpha must be fp32 with p1's shape and strides")
    dp1, dp2, dv = _like(p1), _like(p1), _like(p1)
    dalpha = _like(alpha)
    need = linear_bwd_workspace_size(p1, kernel)
    if workspace is None:
        workspace = torch.empty(max(need, 16), device=p1.device, dtype=torch.uint8)
    rc = load().relation_linear_bwd_ex(_ptr(p1), _ptr(p2), _ptr(v), _ptr(alpha), _ptr(dy),
                                       _ptr(dp1), _ptr(dp2), _ptr(dv), _ptr(dalpha),
                                       float(tau_s), shape_of(p1), _dtype_code(p1),
                                       KERNELS[kernel], _ptr(workspace),
                                       workspace.numel() * workspace.element_size(),
                                       _ptr(dev_status), ctypes.c_void_p(_stream(stream)))
    if rc != OK:
        raise RelationError(rc, "relation_linear_bwd_ex")
    return dp1, dp2, dv, dalpha


def _layer_args(theta, pairing, rope_base, x):
    if theta.dtype != torch.float32 or theta.device != x.device or theta.numel() != x.shape[2] // 2:
        raise ValueError("theta must be fp32 [H/2] on the inputs' device")
    if pairing not in (0, 1):
        raise ValueError("pairing must be 0 (pairs (0,1), (2,3), ...) or 1 ((1,2), ..., (H-1,0))")
    return theta.contiguous(), int(pairing), float(rope_base)


def layer_prep(p1, p2, info, theta, pairing: int = 0, rope_base: float = 1.0e4, *, out=None,
               stream=None):
    """The layer's transforms before the operator: returns (q, k, v) = (RoPE(p1),
    RoPE(p2), Givens(info)) for [B, T, H, d] inputs of one layout, theta fp32 [H/2]."""
    _same_layout(p1, p2, info)
    theta, pairing, rope_base = _layer_args(theta, pairing, rope_base, p1)
    q, k, v = out if out is not None else (_like(p1), _like(p1),
                                           _like(p1))
    _same_layout(p1, q, k, v)
    rc = load().relation_layer_prep(_ptr(p1), _ptr(p2), _ptr(info), _ptr(theta), pairing,
                                    rope_base, _ptr(q), _ptr(k), _ptr(v), shape_of(p1),
                                    _dtype_code(p1), ctypes.c_void_p(_stream(stream)))
    if rc != OK:
        raise RelationError(rc, "relation_layer_prep")
    return q, k, v


def layer_grad_workspace_size(x) -> int:
    """Device bytes relation_layer_grad needs for a [B, T, H, d] tensor of this dtype."""
    return int(load().relation_layer_grad_workspace_size(shape_of(x), _dtype_code(x)))


def layer_grad(dq, dk, dv, info, theta, pairing: int = 0, rope_base: float = 1.0e4, *,
               workspace=None, stream=None):
    """Gradient of layer_prep: returns (dp1, dp2, dinfo, dtheta)."""
    _same_layout(dq, dk, dv, info)
    theta, pairing, rope_base = _layer_args(theta, pairing, rope_base, dq)
    dp1, dp2, dinfo = _like(dq), _like(dq), _like(dq)
    dtheta = _like(theta)
    need = layer_grad_workspace_size(dq)
    if workspace is None:
        workspace = torch.empty(max(need, 16), device=dq.device, dtype=torch.uint8)
    rc = load().relation_layer_grad(_ptr(dq), _ptr(dk), _ptr(dv), _ptr(info), _ptr(theta),
                                    pairing, rope_base, _ptr(dp1), _ptr(dp2), _ptr(dinfo),
                                    _ptr(dtheta), shape_of(dq), _dtype_code(dq), _ptr(workspace),
                                    workspace.numel() * workspace.element_size(),
                                    ctypes.c_void_p(_stream(stream)))
    if rc != OK:
        raise RelationError(rc, "relation_layer_grad")
    return dp1, dp2, dinfo, dtheta


def decode_workspace_size(k_cache) -> int:
    """Device bytes relation_decode needs for a [B, T, H, d] cache of this dtype."""
    return int(load().relation_decode_workspace_size(shape_of(k_cache), _dtype_code(k_cache)))


def decode(q, k_cache, v_cache, lengths, lam: float, tau_s: float = 2.0, *, out=None, logz=None,
           workspace=None, dev_status=None, stream=None):
    """One new token per sequence against a [B, T, H, d] key/value cache whose row
    lengths[b] - 1 is that token.  q is [B, H, d]; lengths is a device int32 [B].
    Returns (Y [B, H, d], logZ [B, H])."""
    _same_layout(k_cache, v_cache)
    B, T, H, d = k_cache.shape
    if tuple(q.shape) != (B, H, d) or q.stride(2) != 1 or q.dtype != k_cache.dtype:
        raise ValueError("q must be [B, H, d] with d contiguous, of the cache's dtype")
    if lengths.dtype != torch.int32 or lengths.numel() != B or not lengths.is_contiguous():
        raise ValueError("lengths must be a contiguous int32 tensor of B entries")
    out = _like(q) if out is None else out
    if tuple(out.stride()) != tuple(q.stride()):
        raise ValueError("out must have q's layout")
    if logz is None:
        logz = torch.empty((B, H), device=q.device, dtype=torch.float32)
    need = decode_workspace_size(k_cache)
    if workspace is None:
        workspace = torch.empty(need, device=q.device, dtype=torch.uint8)
    rc = load().relation_decode(_ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(lengths), _ptr(out),
                                _ptr(logz), float(lam), float(tau_s), shape_of(k_cache),
                                q.stride(0), q.stride(1), _dtype_code(q), _ptr(workspace),
                                workspace.numel() * workspace.element_size(), _ptr(dev_status),
                                ctypes.c_void_p(_stream(stream)))
    if rc != OK:
        raise RelationError(rc, "relation_decode")
    return out, logz


BWD_PREPARE, BWD_TILES, BWD_FINALIZE, BWD_ALL = 1, 2, 4, 7


def bwd(q, k, v, o, dout, logz, lam: float, tau_s: float = 2.0, *, kernel: str = "auto",
        workspace=None, dq=None, dk=None, dv=None, dlambda=None, dev_status=None, stream=None,
        stages: int = BWD_ALL):
    """Backward.  Returns (dQ, dK, dV, dlambda) with dlambda a 1-element fp32 device tensor.
    ``stages`` selects a subset of the three backward stages (see relation_bwd_stages)."""
    _same_layout(q, k, v, o, dout)
    dq = _like(q) if dq is None else dq
    dk = _like(q) if dk is None else dk
    dv = _like(q) if dv is None else dv
    _same_layout(q, dq, dk, dv)
    if dlambda is None:
        dlambda = torch.empty(1, device=q.device, dtype=torch.float32)
    need = workspace_size(q)
    if workspace is None:
        workspace = torch.empty(need, device=q.device, dtype=torch.uint8)
    rc = load().relation_bwd_stages(_ptr(q), _ptr(k), _ptr(v), _ptr(o), _ptr(dout), _ptr(logz),
                                    _ptr(dq), _ptr(dk), _ptr(dv), _ptr(dlambda), float(lam),
                                    float(tau_s), shape_of(q), _dtype_code(q),
                                    _ptr(workspace), workspace.numel() * workspace.element_size(),
                                    KERNELS[kernel], int(stages), _ptr(dev_status),
                                    ctypes.c_void_p(_stream(stream)))
    if rc != OK:
        raise RelationError(rc, "relation_bwd")
    return dq, dk, dv, dlambda


def launches_per_call(kernel: str, dtype: str, d: int, which: str) -> int:
    """Kernel launches one fwd / bwd call makes (0 when unsupported)."""
    dt = F32 if dtype in ("fp32", "f32", torch.float32) else BF16
    return int(load().relation_launch_count(dt, int(d), KERNELS[kernel], int(which == "bwd")))


STATIC_SCRATCH_BYTES = 64 << 20  # RELATION_STATIC_SCRATCH_BYTES


def bwd_no_alloc(q, k, v, o, dout, logz, lam: float, tau_s: float = 2.0, *,
                 kernel: str = "auto", dq, dk, dv, dlambda, dev_status=None, stream=None):
    """Backward through relation_bwd_static: the library's fixed scratch array replaces the
    workspace, for callers that must not allocate device memory.  All outputs are
    caller-provided (this function allocates nothing either)."""
    _same_layout(q, k, v, o, dout, dq, dk, dv)
    rc = load().relation_bwd_static(_ptr(q), _ptr(k), _ptr(v), _ptr(o), _ptr(dout), _ptr(logz),
                                    _ptr(dq), _ptr(dk), _ptr(dv), _ptr(dlambda), float(lam),
                                    float(tau_s), shape_of(q), _dtype_code(q), KERNELS[kernel],
                                    _ptr(dev_status), ctypes.c_void_p(_stream(stream)))
    if rc != OK:
        raise RelationError(rc, "relation_bwd_static")
    return dq, dk, dv, dlambda


def selftest_wait_timeout(dev_status: torch.Tensor, timeout_us: int = 1000, stream=None) -> int:
    """Launch the bounded-wait self-test; returns the launch status."""
    return int(load().relation_selftest_wait_timeout(_ptr(dev_status), int(timeout_us),
                                                     ctypes.c_void_p(_stream(stream))))


class RelationFunction(torch.autograd.Function):
    """Autograd wrapper: Y = Relation(q, k, v; lambda).  lambda is a 1-element tensor
    (its gradient is returned); tau_S is a constant."""

    @staticmethod
    def forward(ctx, q, k, v, lam, tau_s=2.0, kernel="auto"):
        y, logz = fwd(q, k, v, float(lam), tau_s, kernel=kernel)
        ctx.save_for_backward(q, k, v, y, logz)
        ctx.lam, ctx.tau_s, ctx.kernel = float(lam), tau_s, kernel
        return y

    @staticmethod
    def backward(ctx, dy):
        q, k, v, y, logz = ctx.saved_tensors
        if dy.stride() != q.stride() or dy.dtype != q.dtype:
            dy = _like(q).copy_(dy)
        dq, dk, dv, dl = bwd(q, k, v, y, dy, logz, ctx.lam, ctx.tau_s, kernel=ctx.kernel)
        return dq, dk, dv, dl.reshape(()).to(torch.float32), None, None
