"""Shared helpers for the tests: device upload of generated inputs and the
tolerance checks stated for this method (fp64 oracle as the reference)."""
import numpy as np

from oracle import bf16_bits_to_f64

# bf16 layers: relative L2 error <= 5e-3 against the fp64 reference, and max-abs error
# <= 3e-2 * RMS(reference) against the fp64 reference rounded once to bf16 (nearest, ties
# to even: the one rounding the output format imposes on an exact result);
# fp32 layers: max-abs error <= 1e-4 * RMS(reference).
# An fp32 result rounded to bf16 lands on the other side of a rounding midpoint from the
# exact value when the two straddle it; so where the output equals the bf16 rounding of
# a value within relative FP32_PATH_REL of the exact one (far above fp32 accumulation
# error, far below a bf16 ulp of 2^-7), that rounding is the reference for the element.
FP32_PATH_REL = 2.0 ** -16
BF16_REL_L2 = 5e-3
BF16_MAX_ABS_RMS = 3e-2
F32_MAX_ABS_RMS = 1e-4


def to_dev(a, dtype):
    import torch
    if a is None:
        return None
    if dtype == "bf16":
        t = torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16)
    else:
        t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32))
    return t.cuda()


def to_dev_f32(a):
    import torch
    if a is None:
        return None
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).cuda()


def host_f64(a, dtype):
    """Inputs as the oracle reads them (bf16 bits -> exact float64)."""
    if a is None:
        return None
    if dtype == "bf16":
        return bf16_bits_to_f64(a)
    return np.asarray(a, dtype=np.float64)


def out_f64(t):
    import torch
    return t.detach().to(torch.float64).cpu().numpy()


BF16_HALF_ULP = 2.0 ** -8  # half a bf16 ulp, relative to the value


def round_bf16(a):
    """Each float64 rounded to the nearest bfloat16 value (ties to even), as float64."""
    a = np.asarray(a, dtype=np.float64)
    m, e = np.frexp(a)  # a = m 2^e, 0.5 <= |m| < 1: 8 significant bits are m 2^8
    r = np.ldexp(np.rint(m * 256.0), e - 8)
    tiny = np.abs(a) < 2.0 ** -126  # bf16 subnormals: a fixed spacing of 2^-133
    return np.where(tiny, np.rint(a * 2.0 ** 133) * 2.0 ** -133, r)


def errors(got, ref, rounded=None):
    """rel-L2 against ref, max-abs against `rounded` (ref when None), RMS of ref."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    rms = float(np.sqrt(np.mean(ref * ref))) if ref.size else 0.0
    rel_l2 = float(np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-300))
    target = ref if rounded is None else rounded
    max_abs = float(np.abs(got - target).max()) if got.size else 0.0
    return rel_l2, max_abs, rms


def bf16_reference(got, ref):
    """ref rounded to bf16; where got is the rounding of ref * (1 -+ FP32_PATH_REL), that."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    r = round_bf16(ref)
    lo = round_bf16(ref * (1.0 - FP32_PATH_REL))
    hi = round_bf16(ref * (1.0 + FP32_PATH_REL))
    return np.where((got == lo) | (got == hi), got, r)


def assert_bf16_close(got, ref, what=""):
    rel_l2, max_abs, rms = errors(got, ref, bf16_reference(got, ref))
    assert np.isfinite(got).all(), what + ": non-finite output"
    assert rel_l2 <= BF16_REL_L2, "%s: rel-L2 %.3e > %.1e" % (what, rel_l2, BF16_REL_L2)
    assert max_abs <= BF16_MAX_ABS_RMS * rms, "%s: max-abs %.3e > %.1e * RMS %.3e" % (
        what, max_abs, BF16_MAX_ABS_RMS, rms)
    return rel_l2, max_abs, rms


def assert_f32_close(got, ref, what=""):
    rel_l2, max_abs, rms = errors(got, ref)
    assert np.isfinite(got).all(), what + ": non-finite output"
    assert max_abs <= F32_MAX_ABS_RMS * rms, "%s: max-abs %.3e > %.1e * RMS %.3e" % (
        what, max_abs, F32_MAX_ABS_RMS, rms)
    return rel_l2, max_abs, rms
