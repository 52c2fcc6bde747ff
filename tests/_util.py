"""Shared helpers of the GPU parity tests (host-side marshalling only)."""
import numpy as np
import torch

from paper_2111_11581_gb300 import inputs

TOL = 1e-2      # max |err| <= 1e-2 * max(1, |ref|), fp32 accumulation vs fp64 oracle


def dev16(bits: np.ndarray, dtype: int, pad_last_to: int = 1) -> torch.Tensor:
    """uint16 bit patterns -> cuda fp16/bf16 tensor; last dim padded (stride) to a multiple."""
    t = inputs.as_torch(np.ascontiguousarray(bits), dtype)
    if pad_last_to > 1 and t.dim() == 2 and t.shape[1] % pad_last_to:
        n = t.shape[1]
        ld = (n + pad_last_to - 1) // pad_last_to * pad_last_to
        buf = torch.zeros((t.shape[0], ld), dtype=t.dtype)
        buf[:, :n] = t
        return buf.cuda()[:, :n]
    return t.cuda()


def host_bits(t: torch.Tensor) -> np.ndarray:
    return t.detach().contiguous().cpu().view(torch.int16).numpy().view(np.uint16)


def assert_close(got_bits: np.ndarray, ref_bits: np.ndarray, dtype: int, what: str = ""):
    import oracle
    g = oracle.to_double(np.ascontiguousarray(got_bits), dtype)
    r = oracle.to_double(np.ascontiguousarray(ref_bits), dtype)
    assert g.shape == r.shape, (g.shape, r.shape)
    err = np.abs(g - r)
    bound = TOL * np.maximum(1.0, np.abs(r))
    bad = ~(err <= bound)
    if bad.any():
        i = np.argwhere(bad)[0]
        raise AssertionError(f"{what}: {int(bad.sum())} of {bad.size} outside tolerance; first at "
                             f"{tuple(i)} got {g[tuple(i)]} ref {r[tuple(i)]}; "
                             f"max err {err.max():.4g}")
