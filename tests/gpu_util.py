"""Helpers for the GPU parity tests: device copies, the plan factory, and the
comparison rule.

Comparison rule (the acceptance bar of the projection):
* INT32 accumulators: bit-exact against the CPU oracle.
* FP32 outputs: tolerance 1 ulp (``Y_ULP_TOL``); both sides perform one
  correctly rounded FP32 multiply of the same operands, so 0 ulp -- identical
  bits, signed zeros included -- is what the library delivers, and the tests
  require it too (``exact=True``).
"""
from __future__ import annotations

import numpy as np
import torch

DEV = "cuda:0"
Y_ULP_TOL = 1


def to_dev(a: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a)).to(DEV)


def ordered(bits: np.ndarray) -> np.ndarray:
    """FP32 bit patterns -> integers ordered like the floats (+0 == -0)."""
    i = bits.view(np.int32).astype(np.int64)
    return np.where(i < 0, -(i & 0x7FFFFFFF), i)


def ulp_distance(a: np.ndarray, b: np.ndarray) -> np.ndarray:
    return np.abs(ordered(np.asarray(a, np.float32)) - ordered(np.asarray(b, np.float32)))


def assert_parity(acc, y, acc_ref, y_ref, what="", exact=True):
    """acc / y: torch tensors (or numpy) from the GPU; *_ref: oracle numpy."""
    a = acc.detach().cpu().numpy() if hasattr(acc, "detach") else np.asarray(acc)
    a = a.reshape(acc_ref.shape)
    bad = np.argwhere(a != acc_ref)
    assert bad.size == 0, (f"{what}: {len(bad)} INT32 mismatches of {a.size}; first "
                           f"{[(tuple(i), int(a[tuple(i)]), int(acc_ref[tuple(i)])) for i in bad[:4]]}")
    if y is None:
        return
    yy = y.detach().cpu().numpy() if hasattr(y, "detach") else np.asarray(y)
    yy = yy.reshape(y_ref.shape).astype(np.float32)
    d = ulp_distance(yy, y_ref)
    assert d.max(initial=0) <= Y_ULP_TOL, f"{what}: FP32 off by {d.max()} ulp"
    if exact:
        nb = int(np.count_nonzero(yy.view(np.uint32) != y_ref.view(np.uint32)))
        assert nb == 0, f"{what}: {nb} FP32 outputs differ in their bits (0 ulp expected)"
