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


def oracle_experts(seed, experts, hidden, inter, device="cuda"):
    """Oracle-packed blocks of the given experts, from the generator's fp32
    weights (the same draws the GPU layer was packed from)."""
    import oracle
    from paper_2608_08910_gb300 import inputs
    out = {}
    for e in experts:
        out[int(e)] = tuple(
            oracle.pack_rtn(inputs.expert_matrix(seed, int(e), p, hidden, inter, device).cpu().numpy())
            for p in (inputs.PROJ_GATE, inputs.PROJ_UP, inputs.PROJ_DOWN))
    return out


def selection_tolerance(Wr, x, bias):
    """Per-expert bound on |kernel logit - oracle logit|: the kernel's
    compensated binary32 dot product (Dot2, error below gamma_n^2 sum|w x|
    with per-thread chains of n <= H/128 terms, then double-binary32 sums
    with relative error near 2^-44) plus the oracle's sequential binary64
    sum (H 2^-53 sum|w x|), doubled for safety."""
    terms = np.abs(Wr.astype(np.float64)) @ np.abs(x.astype(np.float64))
    H = Wr.shape[1]
    b = 0 if bias is None else np.abs(bias.astype(np.float64))
    gamma = (H // 128 + 2) * 2.0 ** -24
    return 2 * (gamma ** 2 + 16 * 2.0 ** -44 + H * 2.0 ** -53) * (terms + b) + 1e-300


def check_selection(sel, logits, tol, k):
    """Expert ids must equal the oracle's ranking except where two adjacent
    candidates (ranks 0..k) are closer than the error bound. Returns the
    number of accepted near-tie swaps."""
    order = np.lexsort((np.arange(logits.size), -logits))
    ties = 0
    for r in range(k):
        a = order[r]
        b = order[r + 1] if r + 1 < logits.size else order[r]
        close = abs(logits[a] - logits[b]) <= tol[a] + tol[b]
        if sel[r] != order[r]:
            assert close, "rank %d: got expert %d, oracle %d" % (r, sel[r], order[r])
            ties += 1
    return ties
