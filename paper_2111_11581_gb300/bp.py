"""Thin ctypes binding of libbp.so (include/bp.h).

The ``bp_*`` functions mirror the C entry points one to one and take raw
device pointers (ints) and sizes.  The lower-case helpers below them only
allocate outputs with torch and marshal tensors to those calls; every step of
the computation runs in the library's CUDA kernels.  If libbp.so cannot be
loaded, an error is raised: there is no CPU fallback.
"""
from __future__ import annotations

import ctypes
import os
import threading
from dataclasses import dataclass

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libbp.so")

F16, BF16 = 0, 1
BLOCK_BASED, BLOCK_PUNCHED = 0, 1
OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_NONFINITE, ERR_WORKSPACE, ERR_CUDA, ERR_TIMEOUT = range(7)


class Layout(ctypes.Structure):
    _fields_ = [("scheme", ctypes.c_int32), ("dtype", ctypes.c_int32), ("M", ctypes.c_int64),
                ("K", ctypes.c_int64), ("kh", ctypes.c_int32), ("kw", ctypes.c_int32),
                ("bm", ctypes.c_int32), ("bk", ctypes.c_int32)]


class Packed(ctypes.Structure):
    _fields_ = [("lay", Layout), ("num_rb", ctypes.c_int64), ("nnz_cols", ctypes.c_int64),
                ("nnz_vals", ctypes.c_int64), ("rb_ptr", ctypes.c_void_p),
                ("col_idx", ctypes.c_void_p), ("values", ctypes.c_void_p),
                ("dev", ctypes.c_void_p), ("dev_bytes", ctypes.c_int64)]


EXPORTS = ("bp_status_string", "bp_version", "bp_workspace_size", "bp_prune", "bp_prune_rows",
           "bp_prune_pattern",
           "bp_pack_size", "bp_pack", "bp_gemm", "bp_gemm_workspace_size", "bp_conv2d",
           "bp_conv2d_workspace_size", "bp_penalty_units", "bp_reweighted_penalty",
           "bp_penalty_workspace_size", "bp_device_status", "bp_set_watchdog_ns",
           "bp_debug_drop_stage", "bp_prune_noalloc")

_lib = None
_lock = threading.Lock()


class BpError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {status_string(status)} ({status})")


def load(path: str = LIB_PATH):
    """Open libbp.so and declare the signatures (raises if it is missing)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(path):
            raise OSError(f"libbp.so not built ({path}); run paper_2111_11581_gb300.build")
        lib = ctypes.CDLL(path)
        vp, i64, i32, dbl, sz = (ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_double,
                                 ctypes.c_size_t)
        P_L, P_P = ctypes.POINTER(Layout), ctypes.POINTER(Packed)
        P_i64 = ctypes.POINTER(ctypes.c_int64)
        sig = {
            "bp_status_string": (ctypes.c_char_p, [i32]),
            "bp_version": (i32, []),
            "bp_workspace_size": (i32, [P_L, ctypes.POINTER(sz)]),
            "bp_prune": (i32, [P_L, vp, dbl, vp, vp, sz, vp]),
            "bp_prune_rows": (i32, [P_L, vp, dbl, vp, vp, sz, vp]),
            "bp_prune_pattern": (i32, [P_L, vp, dbl, vp, i32, vp, vp, sz, vp]),
            "bp_pack_size": (i32, [P_L, vp, vp, P_i64, P_i64, P_i64, vp]),
            "bp_pack": (i32, [P_L, vp, vp, P_P, vp]),
            "bp_gemm": (i32, [P_P, vp, i64, i64, vp, i32, vp, i64, vp, sz, vp]),
            "bp_gemm_workspace_size": (i32, [P_P, i64, ctypes.POINTER(sz)]),
            "bp_conv2d": (i32, [P_P, vp, i64, i64, i64, i64, i32, i32, i32, i32, vp, i32, vp,
                                vp, sz, vp]),
            "bp_conv2d_workspace_size": (i32, [P_P, i64, i64, i64, i64, i32, i32, i32, i32,
                                               ctypes.POINTER(sz)]),
            "bp_penalty_units": (i32, [P_L, i32, P_i64]),
            "bp_reweighted_penalty": (i32, [P_L, i32, vp, dbl, dbl, vp, vp, vp, vp, sz, vp]),
            "bp_penalty_workspace_size": (i32, [P_L, i32, ctypes.POINTER(sz)]),
            "bp_device_status": (i32, [vp]),
            "bp_set_watchdog_ns": (i32, [ctypes.c_uint64]),
            "bp_debug_drop_stage": (i32, [i64]),
            "bp_prune_noalloc": (i32, [P_L, vp, dbl, vp, vp]),
        }
        for name, (res, args) in sig.items():
            f = getattr(lib, name)
            f.restype, f.argtypes = res, args
        # BP_WATCHDOG_NS: the bound on every kernel wait (bp_set_watchdog_ns),
        # e.g. raised under a profiler that replays each launch many times
        wd = os.environ.get("BP_WATCHDOG_NS")
        if wd:
            lib.bp_set_watchdog_ns(int(float(wd)))
        _lib = lib
        return lib


def status_string(status: int) -> str:
    return load().bp_status_string(int(status)).decode()


def _chk(st: int, what: str):
    if st != OK:
        raise BpError(st, what)


# ------------------------------------------------------------------ C entry points
def bp_version() -> int:
    return load().bp_version()


def bp_workspace_size(lay: Layout) -> int:
    n = ctypes.c_size_t()
    _chk(load().bp_workspace_size(ctypes.byref(lay), ctypes.byref(n)), "bp_workspace_size")
    return n.value


def bp_prune(lay: Layout, W: int, rate: float, mask: int, ws: int, ws_bytes: int,
             stream: int = 0) -> int:
    return load().bp_prune(ctypes.byref(lay), W, float(rate), mask, ws, ws_bytes, stream)


def bp_prune_rows(lay: Layout, W: int, rate: float, mask: int, ws: int, ws_bytes: int,
                  stream: int = 0) -> int:
    return load().bp_prune_rows(ctypes.byref(lay), W, float(rate), mask, ws, ws_bytes, stream)


def bp_prune_pattern(lay: Layout, W: int, rate: float, patterns, mask: int, ws: int,
                     ws_bytes: int, stream: int = 0) -> int:
    pats = (ctypes.c_uint16 * len(patterns))(*[int(p) for p in patterns])
    return load().bp_prune_pattern(ctypes.byref(lay), W, float(rate), pats, len(patterns), mask,
                                   ws, ws_bytes, stream)


def bp_pack_size(lay: Layout, mask: int, rb_ptr: int, stream: int = 0):
    nc, nv, db = ctypes.c_int64(), ctypes.c_int64(), ctypes.c_int64()
    st = load().bp_pack_size(ctypes.byref(lay), mask, rb_ptr, ctypes.byref(nc),
                             ctypes.byref(nv), ctypes.byref(db), stream)
    return st, nc.value, nv.value, db.value


def bp_pack(lay: Layout, W: int, mask: int, packed: Packed, stream: int = 0) -> int:
    return load().bp_pack(ctypes.byref(lay), W, mask, ctypes.byref(packed), stream)


def bp_gemm(packed: Packed, X: int, N: int, ldx: int, bias: int | None, relu: int, Y: int,
            ldy: int, ws: int | None = None, ws_bytes: int = 0, stream: int = 0) -> int:
    return load().bp_gemm(ctypes.byref(packed), X, N, ldx, bias, int(relu), Y, ldy, ws, ws_bytes,
                          stream)


def bp_gemm_workspace_size(packed: Packed, N: int):
    n = ctypes.c_size_t()
    st = load().bp_gemm_workspace_size(ctypes.byref(packed), N, ctypes.byref(n))
    return st, n.value


def bp_conv2d(packed: Packed, x: int, Nb: int, C: int, H: int, W: int, pad_h: int, pad_w: int,
              stride_h: int, stride_w: int, bias: int | None, relu: int, out: int,
              ws: int | None, ws_bytes: int, stream: int = 0) -> int:
    return load().bp_conv2d(ctypes.byref(packed), x, Nb, C, H, W, pad_h, pad_w, stride_h,
                            stride_w, bias, int(relu), out, ws, ws_bytes, stream)


def bp_conv2d_workspace_size(packed: Packed, Nb: int, C: int, H: int, W: int, pad_h: int,
                             pad_w: int, stride_h: int, stride_w: int):
    n = ctypes.c_size_t()
    st = load().bp_conv2d_workspace_size(ctypes.byref(packed), Nb, C, H, W, pad_h, pad_w,
                                         stride_h, stride_w, ctypes.byref(n))
    return st, n.value


GROUPS_LAYOUT, GROUPS_ROWS = 0, 1


def bp_penalty_units(lay: Layout, groups: int = GROUPS_LAYOUT):
    n = ctypes.c_int64()
    st = load().bp_penalty_units(ctypes.byref(lay), int(groups), ctypes.byref(n))
    return st, n.value


def bp_penalty_workspace_size(lay: Layout, groups: int = GROUPS_LAYOUT):
    n = ctypes.c_size_t()
    st = load().bp_penalty_workspace_size(ctypes.byref(lay), int(groups), ctypes.byref(n))
    return st, n.value


def bp_reweighted_penalty(lay: Layout, groups: int, W: int, eps: float, lam: float, alpha: int,
                          R: int, grad: int, ws: int | None, ws_bytes: int,
                          stream: int = 0) -> int:
    return load().bp_reweighted_penalty(ctypes.byref(lay), int(groups), W, float(eps),
                                        float(lam), alpha, R, grad, ws, ws_bytes, stream)


def bp_device_status(stream: int = 0) -> int:
    return load().bp_device_status(stream)


def bp_set_watchdog_ns(ns: int) -> int:
    return load().bp_set_watchdog_ns(int(ns))


def bp_prune_noalloc(lay: Layout, W: int, rate: float, mask: int, stream: int = 0) -> int:
    return load().bp_prune_noalloc(ctypes.byref(lay), W, float(rate), mask, stream)


def bp_debug_drop_stage(stage: int) -> int:
    return load().bp_debug_drop_stage(int(stage))


# ------------------------------------------------------------------ torch marshalling
def _torch():
    import torch
    return torch


def _stream(stream=None) -> int:
    torch = _torch()
    s = stream if stream is not None else torch.cuda.current_stream()
    return int(s.cuda_stream)


def _dt(dtype: int):
    torch = _torch()
    return torch.bfloat16 if dtype == BF16 else torch.float16


def layout(scheme: int, dtype: int, M: int, K: int, bm: int, bk: int, kh: int = 1,
           kw: int = 1) -> Layout:
    return Layout(scheme, dtype, M, K, kh, kw, bm, bk)


def prune(lay: Layout, W, rate: float, stream=None):
    """Mask (uint8 M x K, device) of bp_prune on device weight W."""
    torch = _torch()
    mask = torch.empty((lay.M, lay.K), dtype=torch.uint8, device=W.device)
    nbytes = bp_workspace_size(lay)
    ws = torch.empty(max(nbytes, 256), dtype=torch.uint8, device=W.device)
    _chk(bp_prune(lay, W.data_ptr(), rate, mask.data_ptr(), ws.data_ptr(), nbytes, _stream(stream)),
         "bp_prune")
    return mask


def prune_rows(lay: Layout, W, rate: float, mask=None, stream=None):
    """Row pruning (bp_prune_rows) ANDed into `mask` (a new all-ones mask when
    None); returns the mask."""
    torch = _torch()
    if mask is None:
        mask = torch.ones((lay.M, lay.K), dtype=torch.uint8, device=W.device)
    nbytes = bp_workspace_size(lay)
    ws = torch.empty(max(nbytes, 256), dtype=torch.uint8, device=W.device)
    _chk(bp_prune_rows(lay, W.data_ptr(), rate, mask.data_ptr(), ws.data_ptr(), nbytes,
                       _stream(stream)), "bp_prune_rows")
    return mask


# 4-entry 3x3 kernel patterns (pos = 3i + j): the centre with three edge
# neighbours (four T shapes) and the centre with two adjacent edge neighbours
# and the corner between them (four 2 x 2 squares).
DEFAULT_PATTERNS = (0b000111010, 0b010110010, 0b010111000, 0b010011010,
                    0b000011011, 0b000110110, 0b011011000, 0b110110000)


def prune_pattern(lay: Layout, W, rate: float, patterns=DEFAULT_PATTERNS, stream=None):
    """Mask (uint8 M x K, device) of bp_prune_pattern on a 3x3 weight."""
    torch = _torch()
    mask = torch.empty((lay.M, lay.K), dtype=torch.uint8, device=W.device)
    nbytes = bp_workspace_size(lay)
    ws = torch.empty(max(nbytes, 256), dtype=torch.uint8, device=W.device)
    _chk(bp_prune_pattern(lay, W.data_ptr(), rate, patterns, mask.data_ptr(), ws.data_ptr(),
                          nbytes, _stream(stream)), "bp_prune_pattern")
    return mask


@dataclass
class PackedWeight:
    """bp_packed plus the torch tensors that own its device arrays."""
    c: Packed
    rb_ptr: object
    col_idx: object
    values: object
    dev: object

    @property
    def lay(self) -> Layout:
        return self.c.lay


def pack(lay: Layout, W, mask, stream=None) -> PackedWeight:
    torch = _torch()
    dev = W.device
    RB = -(-lay.M // lay.bm)
    rb_ptr = torch.empty(RB + 1, dtype=torch.int64, device=dev)
    st, nc, nv, db = bp_pack_size(lay, mask.data_ptr(), rb_ptr.data_ptr(), _stream(stream))
    _chk(st, "bp_pack_size")
    col_idx = torch.empty(max(nc, 1), dtype=torch.int32, device=dev)
    values = torch.empty(max(nv, 1), dtype=_dt(lay.dtype), device=dev)
    devbuf = torch.empty(max(db, 16), dtype=torch.uint8, device=dev)
    c = Packed(lay, RB, nc, nv, rb_ptr.data_ptr(), col_idx.data_ptr(), values.data_ptr(),
               devbuf.data_ptr(), db)
    _chk(bp_pack(lay, W.data_ptr(), mask.data_ptr(), c, _stream(stream)), "bp_pack")
    return PackedWeight(c, rb_ptr, col_idx[:nc], values[:nv], devbuf)


def gemm_workspace(pw: PackedWeight, N: int, device="cuda"):
    """Device workspace bp_gemm may use for N columns (None when it splits nothing)."""
    torch = _torch()
    st, n = bp_gemm_workspace_size(pw.c, N)
    _chk(st, "bp_gemm_workspace_size")
    return torch.zeros(n, dtype=torch.uint8, device=device) if n else None


def gemm(pw: PackedWeight, X, bias=None, relu: bool = False, out=None, ws=None, stream=None,
         split: bool = True):
    """Y = act(W_masked @ X + bias) through bp_gemm; X is K x N (device).  `ws` from
    gemm_workspace (allocated here when not given; split=False passes none)."""
    torch = _torch()
    K, N = X.shape
    if out is None:
        ldy = (N + 7) // 8 * 8
        out = torch.empty((pw.lay.M, ldy), dtype=X.dtype, device=X.device)[:, :N]
    if ws is None and split:
        ws = gemm_workspace(pw, N, X.device)
    st = bp_gemm(pw.c, X.data_ptr(), N, X.stride(0), None if bias is None else bias.data_ptr(),
                 int(relu), out.data_ptr(), out.stride(0),
                 None if ws is None else ws.data_ptr(),
                 0 if ws is None else ws.numel() * ws.element_size(), _stream(stream))
    _chk(st, "bp_gemm")
    return out


def conv2d_workspace(pw: PackedWeight, shape, pad=(0, 0), stride=(1, 1), device="cuda"):
    """Device workspace bp_conv2d needs for an NCHW input of `shape` (its im2col matrix)."""
    torch = _torch()
    Nb, C, H, W = shape
    st, n = bp_conv2d_workspace_size(pw.c, Nb, C, H, W, pad[0], pad[1], stride[0], stride[1])
    _chk(st, "bp_conv2d_workspace_size")
    return torch.zeros(max(n, 16), dtype=torch.uint8, device=device)


def conv2d(pw: PackedWeight, x, pad=(0, 0), stride=(1, 1), bias=None, relu: bool = False,
           out=None, ws=None, stream=None):
    """NCHW block-sparse convolution through bp_conv2d (`ws` from conv2d_workspace,
    allocated here when not given)."""
    torch = _torch()
    Nb, C, H, W = x.shape
    lay = pw.lay
    Ho = (H + 2 * pad[0] - lay.kh) // stride[0] + 1
    Wo = (W + 2 * pad[1] - lay.kw) // stride[1] + 1
    if out is None:
        out = torch.empty((Nb, lay.M, Ho, Wo), dtype=x.dtype, device=x.device)
    if ws is None:
        ws = conv2d_workspace(pw, x.shape, pad, stride, x.device)
    st = bp_conv2d(pw.c, x.data_ptr(), Nb, C, H, W, pad[0], pad[1], stride[0], stride[1],
                   None if bias is None else bias.data_ptr(), int(relu), out.data_ptr(),
                   ws.data_ptr(), ws.numel() * ws.element_size(), _stream(stream))
    _chk(st, "bp_conv2d")
    return out


def penalty_workspace(lay: Layout, device="cuda", groups: int = GROUPS_LAYOUT):
    """Zero-filled workspace for bp_reweighted_penalty (reusable: every call
    leaves it zeroed)."""
    torch = _torch()
    st, n = bp_penalty_workspace_size(lay, groups)
    _chk(st, "bp_penalty_workspace_size")
    return torch.zeros(n, dtype=torch.uint8, device=device)


def penalty(lay: Layout, W, eps: float, lam: float, ws=None, out=None, stream=None,
            groups: int = GROUPS_LAYOUT):
    """Reweighted regulariser of a layer (bp_reweighted_penalty): returns
    (alpha fp64 [groups], R fp64 [1], grad fp32 M x K) on W's device.  `out`
    may hold a previous result triple to write into."""
    torch = _torch()
    if out is None:
        st, U = bp_penalty_units(lay, groups)
        _chk(st, "bp_penalty_units")
        out = (torch.empty(U, dtype=torch.float64, device=W.device),
               torch.empty(1, dtype=torch.float64, device=W.device),
               torch.empty((lay.M, lay.K), dtype=torch.float32, device=W.device))
    alpha, R, grad = out
    if ws is None:
        ws = penalty_workspace(lay, W.device, groups)
    st = bp_reweighted_penalty(lay, groups, W.data_ptr(), eps, lam, alpha.data_ptr(),
                               R.data_ptr(), grad.data_ptr(), ws.data_ptr(), ws.numel(),
                               _stream(stream))
    _chk(st, "bp_reweighted_penalty")
    return alpha, R, grad


def device_status(stream=None) -> int:
    return bp_device_status(_stream(stream))
