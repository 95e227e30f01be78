"""ctypes binding of libsa_sketch.so (argument marshalling only).

Every function here has the name of the C entry point it calls (see
``include/sa_sketch.h``).  Torch supplies device memory and the current CUDA
stream; all arithmetic runs in the library's kernels.  If the library is not
built or cannot be loaded, every call raises: there is no CPU fallback.
"""
from __future__ import annotations

import ctypes
import math
import os
from typing import Optional, Tuple

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "libsa_sketch.so")

SA_F32, SA_BF16 = 0, 1
SA_KERNEL_FWD_MAIN, SA_KERNEL_BWD_MAIN, SA_KERNEL_AUX, SA_KERNEL_FWD_LSE, SA_KERNEL_BWD_DQ = 0, 1, 2, 3, 4
STATUS = {0: "SA_OK", 1: "SA_ERR_INVALID_ARG", 2: "SA_ERR_UNSUPPORTED", 3: "SA_ERR_WORKSPACE",
          4: "SA_ERR_CUDA", 5: "SA_ERR_TIMEOUT", 6: "SA_ERR_BAD_SEQLENS"}

_lib = None


class SketchError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {STATUS.get(status, status)} ({sa_status_string(status)})")


def load() -> ctypes.CDLL:
    """Load the CUDA library (raises if it is missing: no fallback exists)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is not built; run `python -c 'import __graft_entry__ as g; g.build()'`")
    lib = ctypes.CDLL(LIB_PATH)
    vp, i32, i64, f32, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_float, ctypes.c_size_t
    lib.sa_workspace_size.argtypes = [i32, i64, i32, i32, i32, i32, i32]
    lib.sa_workspace_size.restype = sz
    lib.sa_sketch_fwd.argtypes = [vp, vp, vp, i32, i64, vp, i32, i32, i32, f32, i32, vp, vp, vp, sz, vp]
    lib.sa_sketch_fwd.restype = i32
    lib.sa_sketch_bwd.argtypes = [vp, vp, vp, i32, i64, vp, i32, i32, i32, f32, i32, vp, vp, vp, vp, vp, vp,
                                  sz, vp]
    lib.sa_sketch_bwd.restype = i32
    lib.sa_get_device_error.argtypes = [vp, vp]
    lib.sa_get_device_error.restype = i32
    lib.sa_status_string.argtypes = [i32]
    lib.sa_status_string.restype = ctypes.c_char_p
    lib.sa_timing_enable.argtypes = [i32]
    lib.sa_timing_enable.restype = i32
    lib.sa_timing_read.argtypes = [i32, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_int64)]
    lib.sa_timing_read.restype = i32
    lib.sa_launch_count.argtypes = []
    lib.sa_launch_count.restype = ctypes.c_uint64
    lib.sa_main_kernel_name.argtypes = [i32, i32, i32, i32]
    lib.sa_main_kernel_name.restype = ctypes.c_char_p
    lib.sa_select_path.argtypes = [i32]
    lib.sa_select_path.restype = i32
    lib.sa_sketch_fwd_per_user.argtypes = lib.sa_sketch_fwd.argtypes
    lib.sa_sketch_fwd_per_user.restype = i32
    lib.sa_sketch_bwd_per_user.argtypes = lib.sa_sketch_bwd.argtypes
    lib.sa_sketch_bwd_per_user.restype = i32
    lib.sa_workspace_size_x.argtypes = [i32, i64, i32, i32, i32, i32, i32]
    lib.sa_workspace_size_x.restype = sz
    lib.sa_sketch_fwd_x.argtypes = [vp, vp, i32, i64, vp, vp, i32, i32, i32, f32, i32, vp, vp, vp, sz, vp]
    lib.sa_sketch_fwd_x.restype = i32
    lib.sa_sketch_bwd_x.argtypes = [vp, vp, i32, i64, vp, vp, i32, i32, i32, f32, i32, vp, vp, vp, vp, vp, vp,
                                    sz, vp]
    lib.sa_sketch_bwd_x.restype = i32
    lib.sa_sketch_fwd_noalloc.argtypes = [vp, vp, vp, i32, i64, vp, i32, i32, i32, f32, i32, vp, vp, vp]
    lib.sa_sketch_fwd_noalloc.restype = i32
    lib.sa_noalloc_scratch_bytes.argtypes = []
    lib.sa_noalloc_scratch_bytes.restype = sz
    lib.sa_noalloc_get_device_error.argtypes = [vp]
    lib.sa_noalloc_get_device_error.restype = i32
    lib.sa_set_wait_limit_ns.argtypes = [ctypes.c_uint64]
    lib.sa_set_wait_limit_ns.restype = i32
    lib.sa_workspace_size_tokenwise.argtypes = [i32, i64, i32, i32, i32, i32, i32]
    lib.sa_workspace_size_tokenwise.restype = sz
    lib.sa_sketch_fwd_tokenwise.argtypes = lib.sa_sketch_fwd.argtypes
    lib.sa_sketch_fwd_tokenwise.restype = i32
    lib.sa_sketch_bwd_tokenwise.argtypes = [vp, vp, vp, i32, i64, vp, i32, i32, i32, f32, i32, vp, vp, vp, vp, vp,
                                            vp, vp, sz, vp]
    lib.sa_sketch_bwd_tokenwise.restype = i32
    lib.sa_step_host_workspace_size.argtypes = [vp, i32, i32, i32, i32, i32, i64]
    lib.sa_step_host_workspace_size.restype = sz
    lib.sa_sketch_step_host.argtypes = [vp, vp, vp, i32, i64, vp, i32, i32, i32, f32, i32, vp, vp, vp, vp, vp, i64,
                                        vp, sz, vp]
    lib.sa_sketch_step_host.restype = i32
    lib.sa_plan_chunks_host.argtypes = [vp, i32, i64, vp, vp]
    lib.sa_plan_chunks_host.restype = i32
    lib.sa_plan_host.argtypes = [vp, i32, i32, i32, i32, vp]
    lib.sa_plan_host.restype = i32
    lib.sa_walk_host.argtypes = [vp, i32, i32, i32, i32, vp, vp, vp, vp, ctypes.c_int64]
    lib.sa_walk_host.restype = i32
    _lib = lib
    return lib


def _dt(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return SA_BF16
    if t.dtype == torch.float32:
        return SA_F32
    raise TypeError(f"unsupported dtype {t.dtype} (bf16 or fp32)")


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(device) -> ctypes.c_void_p:
    return ctypes.c_void_p(torch.cuda.current_stream(device).cuda_stream)


def _check(st: int, where: str):
    if st != 0:
        raise SketchError(st, where)


def _validate(K, V, cu, Q):
    for name, t in (("K", K), ("V", V), ("Q", Q), ("cu_seqlens", cu)):
        if not t.is_cuda:
            raise ValueError(f"{name} must be a CUDA tensor")
        if not t.is_contiguous():
            raise ValueError(f"{name} must be contiguous")
    # Q [H,P,d] (prototypes shared by all users) or [B,H,P,d] (per-user queries, Sec. 3.3)
    shared_ok = Q.dim() == 3 and Q.shape[0] == K.shape[1] and Q.shape[2] == K.shape[2]
    per_user_ok = (Q.dim() == 4 and Q.shape[0] == cu.numel() - 1 and Q.shape[1] == K.shape[1]
                   and Q.shape[3] == K.shape[2])
    if K.dim() != 3 or V.shape != K.shape or not (shared_ok or per_user_ok):
        raise ValueError(f"shapes K{tuple(K.shape)} V{tuple(V.shape)} Q{tuple(Q.shape)}: want K,V [N,H,d], "
                         "Q [H,P,d] or [B,H,P,d]")
    if K.dtype != V.dtype or K.dtype != Q.dtype:
        raise ValueError("K, V and Q must share one dtype")
    if cu.dtype != torch.int32 or cu.dim() != 1 or cu.numel() < 2:
        raise ValueError("cu_seqlens must be int32 [B+1]")


# ------------------------------------------------------------- C entry points

def sa_workspace_size(B: int, N: int, H: int, P: int, d: int, dt: int, bwd: bool) -> int:
    return int(load().sa_workspace_size(B, N, H, P, d, dt, int(bool(bwd))))


def sa_status_string(status: int) -> str:
    return load().sa_status_string(status).decode()


def sa_main_kernel_name(P: int, d: int, dt: int, bwd: bool) -> str:
    return load().sa_main_kernel_name(P, d, dt, int(bool(bwd))).decode()


def sa_launch_count() -> int:
    return int(load().sa_launch_count())


def sa_select_path(path: int) -> None:
    """0: tensor-core kernels where supported (default); 1: CUDA cores only;
    2: tensor cores with the lse pass + prototype slices for P = 512."""
    _check(load().sa_select_path(int(path)), "sa_select_path")


def sa_timing_enable(on: bool) -> None:
    _check(load().sa_timing_enable(int(bool(on))), "sa_timing_enable")


def sa_timing_read(kernel_class: int) -> Tuple[float, int]:
    ms, n = ctypes.c_double(), ctypes.c_int64()
    _check(load().sa_timing_read(kernel_class, ctypes.byref(ms), ctypes.byref(n)), "sa_timing_read")
    return ms.value, n.value


def sa_get_device_error(workspace: torch.Tensor) -> int:
    return int(load().sa_get_device_error(_ptr(workspace), _stream(workspace.device)))


_ws_cache = {}


def workspace(nbytes: int, device) -> torch.Tensor:
    """A cached uint8 device buffer of at least ``nbytes`` (allocated by torch)."""
    dev = torch.device(device)
    key = (dev.type, dev.index if dev.index is not None else torch.cuda.current_device())
    buf = _ws_cache.get(key)
    if buf is None or buf.numel() < nbytes:
        buf = torch.empty(max(nbytes, 256), dtype=torch.uint8, device=dev)
        _ws_cache[key] = buf
    return buf


def sa_sketch_fwd(K: torch.Tensor, V: torch.Tensor, cu_seqlens: torch.Tensor, Q: torch.Tensor,
                  scale: Optional[float] = None, want_lse: bool = False,
                  out: Optional[torch.Tensor] = None, lse_out: Optional[torch.Tensor] = None,
                  ws: Optional[torch.Tensor] = None):
    """sketch [B,H,P,d] fp32 (and lse [N,H] fp32 when ``want_lse``).  Q is
    [H,P,d] (C: sa_sketch_fwd) or per user [B,H,P,d] (C: sa_sketch_fwd_per_user)."""
    lib = load()
    _validate(K, V, cu_seqlens, Q)
    N, H, d = K.shape
    P = Q.shape[-2]
    entry = lib.sa_sketch_fwd_per_user if Q.dim() == 4 else lib.sa_sketch_fwd
    B = cu_seqlens.numel() - 1
    dt = _dt(K)
    scale = 1.0 / math.sqrt(d) if scale is None else float(scale)
    sketch = out if out is not None else torch.empty((B, H, P, d), dtype=torch.float32, device=K.device)
    lse = lse_out if lse_out is not None else (
        torch.empty((N, H), dtype=torch.float32, device=K.device) if want_lse else None)
    need = lib.sa_workspace_size(B, N, H, P, d, dt, 0)
    if need == 0:
        raise SketchError(2, "sa_workspace_size")
    w = ws if ws is not None else workspace(need, K.device)
    st = entry(_ptr(K), _ptr(V), _ptr(cu_seqlens), B, N, _ptr(Q), H, P, d, scale, dt,
               _ptr(sketch), _ptr(lse), _ptr(w), w.numel(), _stream(K.device))
    _check(st, "sa_sketch_fwd_per_user" if Q.dim() == 4 else "sa_sketch_fwd")
    return (sketch, lse) if want_lse or lse_out is not None else sketch


def sa_sketch_bwd(K: torch.Tensor, V: torch.Tensor, cu_seqlens: torch.Tensor, Q: torch.Tensor,
                  dsketch: torch.Tensor, scale: Optional[float] = None,
                  lse: Optional[torch.Tensor] = None, outs=None, ws: Optional[torch.Tensor] = None):
    """(dK, dV, dQ): dK, dV like K; dQ fp32 shaped like Q ([H,P,d] summed over
    users, or [B,H,P,d] per user: C sa_sketch_bwd / sa_sketch_bwd_per_user)."""
    lib = load()
    _validate(K, V, cu_seqlens, Q)
    N, H, d = K.shape
    P = Q.shape[-2]
    entry = lib.sa_sketch_bwd_per_user if Q.dim() == 4 else lib.sa_sketch_bwd
    B = cu_seqlens.numel() - 1
    if dsketch.shape != (B, H, P, d) or dsketch.dtype != torch.float32 or not dsketch.is_contiguous():
        raise ValueError("dsketch must be contiguous fp32 [B,H,P,d]")
    if lse is not None and (lse.shape != (N, H) or lse.dtype != torch.float32 or not lse.is_contiguous()):
        raise ValueError("lse must be contiguous fp32 [N,H]")
    dt = _dt(K)
    scale = 1.0 / math.sqrt(d) if scale is None else float(scale)
    if outs is None:
        dK, dV = torch.empty_like(K), torch.empty_like(V)
        dQ = torch.empty(tuple(Q.shape), dtype=torch.float32, device=K.device)
    else:
        dK, dV, dQ = outs
    need = lib.sa_workspace_size(B, N, H, P, d, dt, 1)
    if need == 0:
        raise SketchError(2, "sa_workspace_size")
    w = ws if ws is not None else workspace(need, K.device)
    st = entry(_ptr(K), _ptr(V), _ptr(cu_seqlens), B, N, _ptr(Q), H, P, d, scale, dt,
               _ptr(dsketch), _ptr(lse), _ptr(dK), _ptr(dV), _ptr(dQ), _ptr(w), w.numel(), _stream(K.device))
    _check(st, "sa_sketch_bwd_per_user" if Q.dim() == 4 else "sa_sketch_bwd")
    return dK, dV, dQ


def sa_sketch_fwd_per_user(K, V, cu_seqlens, Q, scale=None, **kw):
    """Forward with per-user queries Q [B,H,P,d] (stacked refinement, Sec. 3.3)."""
    if Q.dim() != 4:
        raise ValueError("per-user queries are [B,H,P,d]")
    return sa_sketch_fwd(K, V, cu_seqlens, Q, scale, **kw)


def sa_sketch_bwd_per_user(K, V, cu_seqlens, Q, dsketch, scale=None, **kw):
    """Backward with per-user queries: dQ [B,H,P,d], each user's own gradient."""
    if Q.dim() != 4:
        raise ValueError("per-user queries are [B,H,P,d]")
    return sa_sketch_bwd(K, V, cu_seqlens, Q, dsketch, scale, **kw)


def sa_sketch_fwd_noalloc(K: torch.Tensor, V: torch.Tensor, cu_seqlens: torch.Tensor, Q: torch.Tensor,
                          scale: Optional[float] = None, out: Optional[torch.Tensor] = None,
                          lse_out: Optional[torch.Tensor] = None):
    """Forward without a workspace: for callers that may not allocate device
    memory when they run this (the library's fixed scratch array is used; see
    include/sa_sketch.h).  ``out`` and ``lse_out`` are the caller's buffers;
    when they are not given they are created here, before the call."""
    lib = load()
    _validate(K, V, cu_seqlens, Q)
    N, H, d = K.shape
    if Q.dim() != 3:
        raise ValueError("sa_sketch_fwd_noalloc takes shared prototypes Q [H,P,d]")
    P = Q.shape[1]
    B = cu_seqlens.numel() - 1
    scale = 1.0 / math.sqrt(d) if scale is None else float(scale)
    sketch = out if out is not None else torch.empty((B, H, P, d), dtype=torch.float32, device=K.device)
    # the library uses the fixed array of the CURRENT device: make K's device current
    with torch.cuda.device(K.device):
        st = lib.sa_sketch_fwd_noalloc(_ptr(K), _ptr(V), _ptr(cu_seqlens), B, N, _ptr(Q), H, P, d, scale,
                                       _dt(K), _ptr(sketch), _ptr(lse_out), _stream(K.device))
    _check(st, "sa_sketch_fwd_noalloc")
    return sketch


def sa_noalloc_get_device_error(device=None) -> int:
    """Device-detected status of the last sa_sketch_fwd_noalloc call on
    ``device`` (synchronises its current stream)."""
    device = torch.device("cuda", torch.cuda.current_device()) if device is None else torch.device(device)
    with torch.cuda.device(device):
        return int(load().sa_noalloc_get_device_error(_stream(device)))


def sa_set_wait_limit_ns(ns: int) -> None:
    """Limit of the kernels' bounded pipeline waits for later calls (0 = the
    default 2 s); a test hook for the timeout path."""
    _check(load().sa_set_wait_limit_ns(int(ns)), "sa_set_wait_limit_ns")


def _validate_x(X, cu, Q, Wk):
    for name, t in (("X", X), ("Q", Q), ("Wk", Wk), ("cu_seqlens", cu)):
        if not t.is_cuda or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous CUDA tensor")
    N, H, d = X.shape
    if Q.dim() != 3 or Q.shape[0] != H or Q.shape[2] != d or tuple(Wk.shape) != (H, d, d):
        raise ValueError(f"shapes X{tuple(X.shape)} Q{tuple(Q.shape)} Wk{tuple(Wk.shape)}: "
                         "want X [N,H,d], Q [H,P,d], Wk [H,d,d]")
    if X.dtype != Q.dtype or X.dtype != Wk.dtype:
        raise ValueError("X, Q and Wk must share one dtype")
    if cu.dtype != torch.int32 or cu.dim() != 1 or cu.numel() < 2:
        raise ValueError("cu_seqlens must be int32 [B+1]")


def sa_sketch_fwd_x(X: torch.Tensor, cu_seqlens: torch.Tensor, Q: torch.Tensor, Wk: torch.Tensor,
                    scale: Optional[float] = None, want_lse: bool = False, ws: Optional[torch.Tensor] = None):
    """Sketch with keys X Wk[h] and values X (Sec. 3.1): [B,H,P,d] fp32 (and lse)."""
    lib = load()
    _validate_x(X, cu_seqlens, Q, Wk)
    N, H, d = X.shape
    P = Q.shape[1]
    B = cu_seqlens.numel() - 1
    dt = _dt(X)
    scale = 1.0 / math.sqrt(d) if scale is None else float(scale)
    sketch = torch.empty((B, H, P, d), dtype=torch.float32, device=X.device)
    lse = torch.empty((N, H), dtype=torch.float32, device=X.device) if want_lse else None
    need = lib.sa_workspace_size_x(B, N, H, P, d, dt, 0)
    if need == 0:
        raise SketchError(2, "sa_workspace_size_x")
    w = ws if ws is not None else workspace(need, X.device)
    st = lib.sa_sketch_fwd_x(_ptr(X), _ptr(cu_seqlens), B, N, _ptr(Q), _ptr(Wk), H, P, d, scale, dt,
                             _ptr(sketch), _ptr(lse), _ptr(w), w.numel(), _stream(X.device))
    _check(st, "sa_sketch_fwd_x")
    return (sketch, lse) if want_lse else sketch


def sa_sketch_bwd_x(X: torch.Tensor, cu_seqlens: torch.Tensor, Q: torch.Tensor, Wk: torch.Tensor,
                    dsketch: torch.Tensor, scale: Optional[float] = None, lse: Optional[torch.Tensor] = None,
                    ws: Optional[torch.Tensor] = None):
    """(dX like X, dQ [H,P,d] fp32, dWk [H,d,d] fp32) for ``sa_sketch_fwd_x``."""
    lib = load()
    _validate_x(X, cu_seqlens, Q, Wk)
    N, H, d = X.shape
    P = Q.shape[1]
    B = cu_seqlens.numel() - 1
    if dsketch.shape != (B, H, P, d) or dsketch.dtype != torch.float32 or not dsketch.is_contiguous():
        raise ValueError("dsketch must be contiguous fp32 [B,H,P,d]")
    dt = _dt(X)
    scale = 1.0 / math.sqrt(d) if scale is None else float(scale)
    dX = torch.empty_like(X)
    dQ = torch.empty((H, P, d), dtype=torch.float32, device=X.device)
    dWk = torch.empty((H, d, d), dtype=torch.float32, device=X.device)
    need = lib.sa_workspace_size_x(B, N, H, P, d, dt, 1)
    if need == 0:
        raise SketchError(2, "sa_workspace_size_x")
    w = ws if ws is not None else workspace(need, X.device)
    st = lib.sa_sketch_bwd_x(_ptr(X), _ptr(cu_seqlens), B, N, _ptr(Q), _ptr(Wk), H, P, d, scale, dt,
                             _ptr(dsketch), _ptr(lse), _ptr(dX), _ptr(dQ), _ptr(dWk), _ptr(w), w.numel(),
                             _stream(X.device))
    _check(st, "sa_sketch_bwd_x")
    return dX, dQ, dWk


def sa_sketch_fwd_tokenwise(K: torch.Tensor, V: torch.Tensor, cu_seqlens: torch.Tensor, Q: torch.Tensor,
                            scale: Optional[float] = None, want_lse: bool = False,
                            ws: Optional[torch.Tensor] = None):
    """Token-wise normalisation (Sec. 5.1, App. C): sketch [B,H,P,d] fp32 with
    weights softmax over each user's tokens per prototype (and lse_tok [B,H,P])."""
    lib = load()
    _validate(K, V, cu_seqlens, Q)
    if Q.dim() != 3:
        raise ValueError("the token-wise variant takes shared prototypes Q [H,P,d]")
    N, H, d = K.shape
    P = Q.shape[1]
    B = cu_seqlens.numel() - 1
    dt = _dt(K)
    scale = 1.0 / math.sqrt(d) if scale is None else float(scale)
    sketch = torch.empty((B, H, P, d), dtype=torch.float32, device=K.device)
    lse = torch.empty((B, H, P), dtype=torch.float32, device=K.device) if want_lse else None
    need = lib.sa_workspace_size_tokenwise(B, N, H, P, d, dt, 0)
    if need == 0:
        raise SketchError(2, "sa_workspace_size_tokenwise")
    w = ws if ws is not None else workspace(need, K.device)
    st = lib.sa_sketch_fwd_tokenwise(_ptr(K), _ptr(V), _ptr(cu_seqlens), B, N, _ptr(Q), H, P, d, scale, dt,
                                     _ptr(sketch), _ptr(lse), _ptr(w), w.numel(), _stream(K.device))
    _check(st, "sa_sketch_fwd_tokenwise")
    return (sketch, lse) if want_lse else sketch


def sa_sketch_bwd_tokenwise(K: torch.Tensor, V: torch.Tensor, cu_seqlens: torch.Tensor, Q: torch.Tensor,
                            dsketch: torch.Tensor, scale: Optional[float] = None,
                            sketch: Optional[torch.Tensor] = None, lse: Optional[torch.Tensor] = None,
                            ws: Optional[torch.Tensor] = None):
    """(dK, dV, dQ [H,P,d] fp32) of ``sa_sketch_fwd_tokenwise``; ``sketch`` and
    ``lse`` are the forward's outputs (recomputed when either is missing)."""
    lib = load()
    _validate(K, V, cu_seqlens, Q)
    if Q.dim() != 3:
        raise ValueError("the token-wise variant takes shared prototypes Q [H,P,d]")
    N, H, d = K.shape
    P = Q.shape[1]
    B = cu_seqlens.numel() - 1
    for name, t, shape in (("dsketch", dsketch, (B, H, P, d)), ("sketch", sketch, (B, H, P, d)),
                           ("lse", lse, (B, H, P))):
        if t is not None and (tuple(t.shape) != shape or t.dtype != torch.float32 or not t.is_contiguous()):
            raise ValueError(f"{name} must be contiguous fp32 {list(shape)}")
    dt = _dt(K)
    scale = 1.0 / math.sqrt(d) if scale is None else float(scale)
    dK, dV = torch.empty_like(K), torch.empty_like(V)
    dQ = torch.empty((H, P, d), dtype=torch.float32, device=K.device)
    need = lib.sa_workspace_size_tokenwise(B, N, H, P, d, dt, 1)
    if need == 0:
        raise SketchError(2, "sa_workspace_size_tokenwise")
    w = ws if ws is not None else workspace(need, K.device)
    st = lib.sa_sketch_bwd_tokenwise(_ptr(K), _ptr(V), _ptr(cu_seqlens), B, N, _ptr(Q), H, P, d, scale, dt,
                                     _ptr(sketch), _ptr(lse), _ptr(dsketch), _ptr(dK), _ptr(dV), _ptr(dQ),
                                     _ptr(w), w.numel(), _stream(K.device))
    _check(st, "sa_sketch_bwd_tokenwise")
    return dK, dV, dQ


def sa_sketch_step_host(K: torch.Tensor, V: torch.Tensor, cu_seqlens: torch.Tensor, Q: torch.Tensor,
                        dsketch: torch.Tensor, scale: Optional[float] = None, chunk_tokens: int = 0,
                        outs=None, device=None, ws: Optional[torch.Tensor] = None):
    """Forward + backward of a batch held in host memory (C: sa_sketch_step_host):
    K, V [N,H,d], cu_seqlens [B+1] int32, Q [H,P,d], dsketch [B,H,P,d] fp32, all
    CPU tensors (page-locked for overlapped copies).  Returns CPU tensors
    (sketch, dK, dV, dQ), written once the current stream of ``device`` is
    synchronised (this function synchronises it before returning)."""
    lib = load()
    for name, t in (("K", K), ("V", V), ("Q", Q), ("cu_seqlens", cu_seqlens), ("dsketch", dsketch)):
        if t.is_cuda or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous CPU tensor")
    N, H, d = K.shape
    P = Q.shape[1]
    B = cu_seqlens.numel() - 1
    if cu_seqlens.dtype != torch.int32 or V.shape != K.shape or tuple(Q.shape) != (H, P, d) or \
            tuple(dsketch.shape) != (B, H, P, d) or dsketch.dtype != torch.float32:
        raise ValueError("shapes: K,V [N,H,d], Q [H,P,d], cu_seqlens int32 [B+1], dsketch fp32 [B,H,P,d]")
    dt = _dt(K)
    scale = 1.0 / math.sqrt(d) if scale is None else float(scale)
    dev = torch.device("cuda", torch.cuda.current_device()) if device is None else torch.device(device)
    if outs is None:
        pin = K.is_pinned()
        outs = (torch.empty((B, H, P, d), dtype=torch.float32, pin_memory=pin),
                torch.empty_like(K, pin_memory=pin), torch.empty_like(V, pin_memory=pin),
                torch.empty((H, P, d), dtype=torch.float32, pin_memory=pin))
    sketch, dK, dV, dQ = outs
    need = lib.sa_step_host_workspace_size(_ptr(cu_seqlens), B, H, P, d, dt, int(chunk_tokens))
    if need == 0:
        raise SketchError(2, "sa_step_host_workspace_size")
    w = ws if ws is not None else workspace(need, dev)
    st = lib.sa_sketch_step_host(_ptr(K), _ptr(V), _ptr(cu_seqlens), B, N, _ptr(Q), H, P, d, scale, dt,
                                 _ptr(dsketch), _ptr(sketch), _ptr(dK), _ptr(dV), _ptr(dQ), int(chunk_tokens),
                                 _ptr(w), w.numel(), _stream(dev))
    _check(st, "sa_sketch_step_host")
    torch.cuda.current_stream(dev).synchronize()
    return sketch, dK, dV, dQ


def sa_plan_chunks_host(cu_seqlens_host, chunk_tokens: int = 0):
    """Chunk boundaries (user indices) sa_sketch_step_host uses (pure C; no GPU)."""
    import numpy as np

    cu = np.ascontiguousarray(cu_seqlens_host, dtype=np.int32)
    begin = np.zeros(cu.size, dtype=np.int32)
    n = ctypes.c_int()
    st = load().sa_plan_chunks_host(cu.ctypes.data, cu.size - 1, int(chunk_tokens), begin.ctypes.data,
                                    ctypes.byref(n))
    _check(st, "sa_plan_chunks_host")
    return begin[: n.value + 1]


def sa_noalloc_scratch_bytes() -> int:
    return int(load().sa_noalloc_scratch_bytes())


def sa_plan_host(cu_seqlens_host, H: int, tile: int, n_workers: int):
    """Host copy of the tiling every call applies (pure C; no GPU)."""
    import numpy as np

    cu = np.ascontiguousarray(cu_seqlens_host, dtype=np.int32)
    begin = np.zeros(n_workers + 1, dtype=np.int64)
    st = load().sa_plan_host(cu.ctypes.data, cu.size - 1, H, tile, n_workers, begin.ctypes.data)
    _check(st, "sa_plan_host")
    return begin


# ------------------------------------------------------------------ autograd

class SketchAttention(torch.autograd.Function):
    """sketch = softmax_proto(scale Q K^T) V per user and head (Sec. 3.1)."""

    @staticmethod
    def forward(ctx, K, V, cu_seqlens, Q, scale):
        sketch, lse = sa_sketch_fwd(K, V, cu_seqlens, Q, scale, want_lse=True)
        ctx.save_for_backward(K, V, cu_seqlens, Q, lse)
        ctx.scale = scale
        return sketch

    @staticmethod
    def backward(ctx, dsketch):
        K, V, cu, Q, lse = ctx.saved_tensors
        dK, dV, dQ = sa_sketch_bwd(K, V, cu, Q, dsketch.contiguous(), ctx.scale, lse=lse)
        return dK, dV, None, dQ.to(Q.dtype), None


def sa_walk_host(cu_seqlens_host, H: int, tile: int, n_workers: int):
    """(user, head, tok0, ntok) of every tile in the order the kernels' workers
    walk them (C: sa_walk_host; pure C, no GPU)."""
    import numpy as np

    cu = np.ascontiguousarray(cu_seqlens_host, dtype=np.int32)
    L = np.diff(cu.astype(np.int64))
    total = int(np.sum((np.maximum(L, 0) + tile - 1) // tile)) * H
    out = (np.zeros(max(total, 1), np.int32), np.zeros(max(total, 1), np.int32), np.zeros(max(total, 1), np.int64),
           np.zeros(max(total, 1), np.int32))
    st = load().sa_walk_host(cu.ctypes.data, cu.size - 1, H, tile, n_workers, *(o.ctypes.data for o in out),
                             max(total, 1))
    _check(st, "sa_walk_host")
    return tuple(o[:total] for o in out)


def sa_sketch(K, V, cu_seqlens, Q, scale: Optional[float] = None):
    """Differentiable sketch [B,H,P,d] (fp32) of packed ragged histories."""
    scale = 1.0 / math.sqrt(K.shape[-1]) if scale is None else float(scale)
    return SketchAttention.apply(K, V, cu_seqlens, Q, scale)
