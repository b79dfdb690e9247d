"""Shared helpers of the test suite (no method arithmetic here)."""
import numpy as np

# Tolerances: max |gpu - ref| / max |ref| over one state tensor or one y block
# (the paper bounds the discrepancy relative to ||h||, Appendix A floating-point note).
TOL_F32 = 1e-5     # fp32 inputs, fp32 state
TOL_BF16 = 2e-3    # bf16 inputs, fp32 state (bf16 storage of the output rounds once: 2^-9)


def rel_err(got, ref) -> float:
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    scale = float(np.max(np.abs(ref))) if ref.size else 0.0
    diff = float(np.max(np.abs(got - ref))) if ref.size else 0.0
    if scale == 0.0:
        return diff
    return diff / scale


def rel_err_stored(got, ref) -> float:
    """rel_err for an output stored in bf16: the tolerance applies to the fp32 value
    before its single rounding to bf16, so each element may additionally differ from the
    reference by half a bf16 ulp of the stored value (round to nearest even)."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    if not ref.size:
        return 0.0
    _, e = np.frexp(got)                       # got = m * 2^e, 0.5 <= |m| < 1
    half_ulp = np.where(got != 0, np.ldexp(1.0, e - 9), 0.0)   # bf16: 8 significant bits
    excess = np.maximum(np.abs(got - ref) - half_ulp, 0.0)
    scale = float(np.max(np.abs(ref)))
    return float(np.max(excess)) / scale if scale else float(np.max(excess))


def to_np(t):
    return t.detach().double().cpu().numpy()
