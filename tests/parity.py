"""Shared helpers of the GPU parity tests (comparison metrics only)."""
import numpy as np


def rel_err(y, ref):
    """max_i |y_i - ref_i| / max(|ref_i|, 1e-3 max_j |ref_j|): the elementwise
    relative error, with a floor that keeps it defined at cancellations."""
    y = np.asarray(y, np.float64)
    ref = np.asarray(ref, np.float64)
    if ref.size == 0:
        return 0.0
    floor = 1e-3 * np.abs(ref).max()
    den = np.maximum(np.abs(ref), floor if floor > 0 else 1e-30)
    return float(np.max(np.abs(y - ref) / den))


FP32_TOL = 1e-4  # the fp32 output bar: max relative error 1e-4
