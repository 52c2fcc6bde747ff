"""CPU oracle for block-based / block-punched pruned-layer inference.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline leg of ``bench.py`` may import this package.  The product
library (``paper_2111_11581_gb300``) never imports it, and it imports nothing
from the product: the two sides share only the seeded input generators.

The arithmetic lives in ``bp_oracle.c`` (plain fp64 loops, compiled with gcc
into ``liboracle.so``); this module marshals numpy arrays to it.  Every
function cites the passage of arXiv 2111.11581 it follows:

* ``scores``          Eq. (column) / Eq. (punched), Sec. 4.2
* ``counts``/``prune`` one-shot magnitude pruning by block, Sec. 4.1 and 5.1
* ``pack``/``unpack``  Blocked Compressed Storage, Sec. 4.3
* ``masked_gemm``      FC / GEMM-view layer with pruned weights skipped, Sec. 4.3
* ``masked_conv2d``    CONV layer (OIHW weight, Sec. 4.2) with pruned weights skipped
* ``to_double``/``round_to``  16-bit float decoding and round-to-nearest-even

Parity of every function is pinned in ``tests/test_oracle.py`` against
brute force, closed forms, special cases and the worked BCS example.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "bp_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

F16, BF16 = 0, 1
BLOCK_BASED, BLOCK_PUNCHED = 0, 1
_ERR = {1: "invalid argument", 3: "non-finite weight"}


def build(force: bool = False) -> str:
    """Compile liboracle.so with gcc (portable flags, OpenMP, no FMA contraction)."""
    if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC):
        return _LIB
    tmp = _LIB + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fopenmp", "-ffp-contract=off", "-fPIC", "-shared",
           _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB)
            i64, i32, dbl, vp = ctypes.c_int64, ctypes.c_int, ctypes.c_double, ctypes.c_void_p
            lib.oracle_half_to_double.restype = dbl
            lib.oracle_half_to_double.argtypes = [ctypes.c_uint16, i32]
            lib.oracle_double_to_half.restype = ctypes.c_uint16
            lib.oracle_double_to_half.argtypes = [dbl, i32]
            lib.oracle_to_double.argtypes = [vp, vp, i64, i32]
            lib.oracle_from_double.argtypes = [vp, vp, i64, i32]
            lib.oracle_num_units.restype = i64
            lib.oracle_num_units.argtypes = [i32, i64, i64, i64, i64, i64, i64]
            lib.oracle_scores.argtypes = [i32, i32, i64, i64, i64, i64, i64, i64, vp, vp]
            lib.oracle_counts.argtypes = [i32, i64, i64, i64, i64, i64, i64, dbl, vp, vp, vp]
            lib.oracle_prune.argtypes = [i32, i32, i64, i64, i64, i64, i64, i64, dbl, vp, vp, vp]
            lib.oracle_pack.argtypes = [i32, i64, i64, i64, vp, vp, vp, vp, vp, vp, vp]
            lib.oracle_unpack.argtypes = [i64, i64, i64, vp, vp, vp, vp, vp]
            lib.oracle_masked_gemm.argtypes = [i32, i64, i64, i64, vp, vp, vp, i64, vp, i32, vp,
                                               i64, vp]
            lib.oracle_masked_conv2d.argtypes = [i32, i64, i64, i64, i64, vp, vp, vp, i64, i64,
                                                 i64, i64, i64, i64, i64, vp, i32, vp, vp]
            lib.oracle_reweighted_penalty.argtypes = [i32, i32, i64, i64, i64, i64, i64, i64, vp,
                                                      dbl, dbl, vp, vp, vp]
            lib.oracle_reweighted_penalty_rows.argtypes = [i32, i64, i64, i64, vp, dbl, dbl, vp,
                                                           vp, vp]
            lib.oracle_prune_rows.argtypes = [i32, i64, i64, i64, i64, dbl, vp, vp, vp]
            lib.oracle_prune_pattern.argtypes = [i32, i64, i64, vp, i32, dbl, vp, vp, vp]
            lib.oracle_max_threads.restype = i32
            for f in ("oracle_scores", "oracle_reweighted_penalty",
                      "oracle_reweighted_penalty_rows", "oracle_counts", "oracle_prune",
                      "oracle_prune_rows", "oracle_prune_pattern",
                      "oracle_pack",
                      "oracle_unpack", "oracle_masked_gemm", "oracle_masked_conv2d"):
                getattr(lib, f).restype = i32
            _lib = lib
    return _lib


class OracleError(RuntimeError):
    pass


def _check(st: int):
    if st != 0:
        raise OracleError(_ERR.get(st, f"status {st}"))


def _p(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _u16(a):
    a = np.ascontiguousarray(a)
    if a.dtype != np.uint16:
        raise TypeError("16-bit float tensors are passed as uint16 bit patterns")
    return a


def max_threads() -> int:
    return int(_load().oracle_max_threads())


def set_threads(n: int) -> None:
    """Threads of the oracle's parallel loops from now on (results do not depend on it)."""
    lib = _load()
    lib.oracle_set_threads.argtypes = [ctypes.c_int]
    lib.oracle_set_threads(int(n))


# ---------------------------------------------------------------- conversions
def to_double(bits, dtype: int) -> np.ndarray:
    """Exact value of each fp16/bf16 bit pattern as float64."""
    b = _u16(bits)
    out = np.empty(b.shape, np.float64)
    _load().oracle_to_double(_p(b), _p(out), b.size, dtype)
    return out


def round_to(x, dtype: int) -> np.ndarray:
    """Round float64 values once to fp16/bf16 (nearest, ties to even); bit patterns."""
    x = np.ascontiguousarray(x, dtype=np.float64)
    out = np.empty(x.shape, np.uint16)
    _load().oracle_from_double(_p(x), _p(out), x.size, dtype)
    return out


# ---------------------------------------------------------------- pruning
def num_units(scheme, M, K, kh, kw, bm, bk) -> int:
    return int(_load().oracle_num_units(scheme, M, K, kh, kw, bm, bk))


def scores(W_bits, dtype, scheme, bm, bk, kh=1, kw=1) -> np.ndarray:
    """Per-unit squared norms, Eq. (column) / Eq. (punched), in unit order g."""
    W = _u16(W_bits)
    M = W.shape[0]
    K = W.size // M
    U = num_units(scheme, M, K, kh, kw, bm, bk)
    if U < 0:
        raise OracleError("invalid argument")
    out = np.empty(U, np.float64)
    _check(_load().oracle_scores(scheme, dtype, M, K, kh, kw, bm, bk, _p(W), _p(out)))
    return out


def reweighted_penalty(W_bits, dtype, scheme, bm, bk, eps, lam, kh=1, kw=1, groups="layout"):
    """Reweighted regulariser of one layer and its gradient (Eq. prob_block with
    Eq. column / Eq. punched, or with Eq. row when groups == "rows"): returns
    (alpha[U], R, grad[M, K]) in fp64."""
    W = _u16(W_bits)
    M, K = W.shape
    if groups == "rows":
        if scheme != 0:
            raise OracleError("row groups are defined for block-based layouts")
        CB = (K + bk - 1) // bk
        alpha = np.zeros(M * CB, np.float64)
        R = np.zeros(1, np.float64)
        grad = np.zeros((M, K), np.float64)
        _check(_load().oracle_reweighted_penalty_rows(dtype, M, K, bk, _p(W), float(eps),
                                                      float(lam), _p(alpha), _p(R), _p(grad)))
        return alpha, float(R[0]), grad
    U = num_units(scheme, M, K, kh, kw, bm, bk)
    alpha = np.zeros(U, np.float64)
    R = np.zeros(1, np.float64)
    grad = np.zeros((M, K), np.float64)
    _check(_load().oracle_reweighted_penalty(scheme, dtype, M, K, kh, kw, bm, bk, _p(W),
                                             float(eps), float(lam), _p(alpha), _p(R), _p(grad)))
    return alpha, float(R[0]), grad


def counts(scheme, M, K, kh, kw, bm, bk, rate):
    """(sum of per-block base counts, total kept units T, global extras E)."""
    sb, T, E = (ctypes.c_int64(), ctypes.c_int64(), ctypes.c_int64())
    _check(_load().oracle_counts(scheme, M, K, kh, kw, bm, bk, float(rate), ctypes.byref(sb),
                                 ctypes.byref(T), ctypes.byref(E)))
    return sb.value, T.value, E.value


def prune(W_bits, dtype, scheme, bm, bk, rate, kh=1, kw=1, return_keep=False):
    """Element mask (M x K uint8) of one-shot block pruning at `rate`."""
    W = _u16(W_bits)
    M = W.shape[0]
    K = W.size // M
    U = num_units(scheme, M, K, kh, kw, bm, bk)
    if U < 0:
        raise OracleError("invalid argument")
    keep = np.empty(U, np.uint8)
    mask = np.empty((M, K), np.uint8)
    _check(_load().oracle_prune(scheme, dtype, M, K, kh, kw, bm, bk, float(rate), _p(W),
                                _p(keep), _p(mask)))
    return (mask, keep) if return_keep else mask


def prune_rows(W_bits, dtype, bm, bk, rate, mask=None, return_keep=False):
    """Row pruning of a block-based layer (rows of each bm x bk block), ANDed
    into `mask` (all ones when None); returns the new M x K uint8 mask (and
    the row-unit flags, numbered block-major then by row)."""
    W = _u16(W_bits)
    M, K = W.shape
    CB = (K + bk - 1) // bk
    m = (np.ones((M, K), np.uint8) if mask is None
         else np.array(mask, dtype=np.uint8, copy=True).reshape(M, K))
    keep = np.empty(M * CB, np.uint8)
    _check(_load().oracle_prune_rows(dtype, M, K, bm, bk, float(rate), _p(W), _p(keep), _p(m)))
    return (m, keep) if return_keep else m


# The 4-entry 3x3 kernel patterns used by default (positions pos = 3i + j):
# the centre with three of its edge neighbours (four "T" shapes) and the
# centre with two adjacent edge neighbours and the corner between them (four
# 2 x 2 squares).
DEFAULT_PATTERNS = np.array([
    (1 << 1) | (1 << 3) | (1 << 4) | (1 << 5),
    (1 << 1) | (1 << 4) | (1 << 5) | (1 << 7),
    (1 << 3) | (1 << 4) | (1 << 5) | (1 << 7),
    (1 << 1) | (1 << 3) | (1 << 4) | (1 << 7),
    (1 << 0) | (1 << 1) | (1 << 3) | (1 << 4),
    (1 << 1) | (1 << 2) | (1 << 4) | (1 << 5),
    (1 << 3) | (1 << 4) | (1 << 6) | (1 << 7),
    (1 << 4) | (1 << 5) | (1 << 7) | (1 << 8),
], np.uint16)


def prune_pattern(W_bits, dtype, rate, patterns=DEFAULT_PATTERNS, return_patterns=False):
    """Pattern-based pruning of an F x C x 3 x 3 weight (kernel patterns +
    connectivity pruning at `rate` >= 9/4): F x 9C uint8 mask (and the chosen
    pattern index of each kernel)."""
    W = _u16(W_bits)
    F = W.shape[0]
    C = W.size // (F * 9)
    pats = np.ascontiguousarray(patterns, np.uint16)
    pat = np.empty(F * C, np.uint8)
    mask = np.empty((F, 9 * C), np.uint8)
    _check(_load().oracle_prune_pattern(dtype, F, C, _p(pats), len(pats), float(rate), _p(W),
                                        _p(pat), _p(mask)))
    return (mask, pat) if return_patterns else mask


def pack(W_bits, mask, bm):
    """Compact storage (rb_ptr int64, col_idx int32, values uint16), Sec. 4.3."""
    W = _u16(W_bits)
    M = W.shape[0]
    K = W.size // M
    m = np.ascontiguousarray(mask, dtype=np.uint8).reshape(M, K)
    nc, nv = ctypes.c_int64(), ctypes.c_int64()
    lib = _load()
    _check(lib.oracle_pack(0, M, K, bm, _p(W), _p(m), None, None, None, ctypes.byref(nc),
                           ctypes.byref(nv)))
    RB = (M + bm - 1) // bm
    rb_ptr = np.empty(RB + 1, np.int64)
    col_idx = np.empty(nc.value, np.int32)
    values = np.empty(nv.value, np.uint16)
    _check(lib.oracle_pack(0, M, K, bm, _p(W), _p(m), _p(rb_ptr), _p(col_idx), _p(values),
                           ctypes.byref(nc), ctypes.byref(nv)))
    return rb_ptr, col_idx, values


def unpack(M, K, bm, rb_ptr, col_idx, values):
    """Dense masked weight (uint16 M x K) and mask from the compact storage."""
    rb_ptr = np.ascontiguousarray(rb_ptr, np.int64)
    col_idx = np.ascontiguousarray(col_idx, np.int32)
    values = _u16(values)
    W = np.empty((M, K), np.uint16)
    mask = np.empty((M, K), np.uint8)
    _check(_load().oracle_unpack(M, K, bm, _p(rb_ptr), _p(col_idx), _p(values), _p(W), _p(mask)))
    return W, mask


# ---------------------------------------------------------------- layer outputs
def masked_gemm(W_bits, mask, X_bits, dtype, bias=None, relu=False, return_acc=False):
    """Y = round(relu(sum_k mask*W*X + bias)), fp64 accumulation, Sec. 4.3."""
    W = _u16(W_bits)
    X = _u16(X_bits)
    M, K = W.shape
    K2, N = X.shape
    if K2 != K:
        raise ValueError("W and X shapes disagree")
    m = np.ascontiguousarray(mask, np.uint8).reshape(M, K)
    b = None if bias is None else np.ascontiguousarray(bias, np.float32)
    Y = np.empty((M, N), np.uint16)
    acc = np.empty((M, N), np.float64) if return_acc else None
    _check(_load().oracle_masked_gemm(dtype, M, K, N, _p(W), _p(m), _p(X), N, _p(b), int(relu),
                                      _p(Y), N, _p(acc)))
    return (Y, acc) if return_acc else Y


def masked_conv2d(W_bits, mask, in_bits, dtype, pad=(0, 0), stride=(1, 1), bias=None,
                  relu=False, return_acc=False):
    """Masked direct convolution (NCHW, OIHW), fp64 accumulation, one rounding."""
    W = _u16(W_bits)
    x = _u16(in_bits)
    F, C, kh, kw = W.shape
    Nb, C2, H, Wd = x.shape
    if C2 != C:
        raise ValueError("channel mismatch")
    m = np.ascontiguousarray(mask, np.uint8).reshape(F, C * kh * kw)
    b = None if bias is None else np.ascontiguousarray(bias, np.float32)
    Ho = (H + 2 * pad[0] - kh) // stride[0] + 1
    Wo = (Wd + 2 * pad[1] - kw) // stride[1] + 1
    out = np.empty((Nb, F, Ho, Wo), np.uint16)
    acc = np.empty((Nb, F, Ho, Wo), np.float64) if return_acc else None
    _check(_load().oracle_masked_conv2d(dtype, F, C, kh, kw, _p(W), _p(m), _p(x), Nb, H, Wd,
                                        pad[0], pad[1], stride[0], stride[1], _p(b), int(relu),
                                        _p(out), _p(acc)))
    return (out, acc) if return_acc else out
