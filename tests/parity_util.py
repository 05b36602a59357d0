"""Tolerances of the parity tests.

fp32 inputs: max-abs error <= 1e-4.  bf16 inputs (fp32 states and
accumulation): max |gpu - ref| / RMS(ref) <= 2e-2, per tensor.  The oracle
always sees the exact (bf16-rounded) values the GPU saw, up-cast to fp64.

A result that the library returns in bf16 carries the rounding of its own
store, up to half a bf16 ulp of the value (2^-9 relative); no computation
can be closer to the fp64 reference than that.  For bf16-typed results the
bound is therefore applied elementwise as
    |gpu - ref| <= 2e-2 * RMS(ref) + ulp_bf16(max(|gpu|, |ref|)) / 2,
and the statistics report the plain max |gpu - ref| / RMS(ref) as well."""
import numpy as np
import torch

TOL_F32_ABS = 1e-4
TOL_BF16_REL = 2e-2
# fp32 states cannot hold magnitudes below the fp32 normal range (1.2e-38;
# the kernels flush denormals), so a tensor whose reference values are all
# that small is compared against this absolute floor instead.
ABS_FLOOR = 1e-35


def as64(t):
    if t is None:
        return None
    if isinstance(t, torch.Tensor):
        return t.detach().float().cpu().double().numpy()
    return np.asarray(t, dtype=np.float64)


def half_ulp_bf16(x):
    """Half the spacing of bf16 numbers at |x| (8 significand bits)."""
    a = np.maximum(np.abs(x), np.finfo(np.float32).tiny)
    return np.exp2(np.floor(np.log2(a)) - 8.0)


def err_stats(gpu, ref):
    g, r = as64(gpu), as64(ref)
    d = np.abs(g - r)
    rms = float(np.sqrt(np.mean(r * r))) if r.size else 0.0
    return dict(max_abs=float(d.max()) if d.size else 0.0, rms_ref=rms,
                max_rel_rms=float(d.max() / rms) if d.size and rms > 0 else 0.0,
                rms_rel=float(np.sqrt(np.mean(d * d)) / rms) if d.size and rms > 0 else 0.0,
                nonfinite=int((~np.isfinite(g)).sum()))


def assert_close(gpu, ref, dtype, name=""):
    s = err_stats(gpu, ref)
    assert s["nonfinite"] == 0, (name, s)
    if dtype == "f32":
        assert s["max_abs"] <= TOL_F32_ABS, (name, s)
        return s
    g, r = as64(gpu), as64(ref)
    bound = TOL_BF16_REL * s["rms_ref"] + ABS_FLOOR
    if isinstance(gpu, torch.Tensor) and gpu.dtype == torch.bfloat16:
        bound = bound + half_ulp_bf16(np.maximum(np.abs(g), np.abs(r)))
    excess = np.abs(g - r) - bound
    assert excess.size == 0 or float(excess.max()) <= 0.0, (name, s)
    return s


def excess_count(gpu, ref):
    """Elements whose error exceeds the plain bound 2e-2 * RMS(ref) (for a
    bf16-typed result these pass only by its half-ulp store rounding)."""
    g, r = as64(gpu), as64(ref)
    rms = float(np.sqrt(np.mean(r * r))) if r.size else 0.0
    return int((np.abs(g - r) > TOL_BF16_REL * rms + ABS_FLOOR).sum())


def record(test, tensor, gpu, ref, **extra):
    """Append one line of error statistics to the file named by the
    RDN_PARITY_REPORT environment variable (nothing when it is unset)."""
    import json
    import os
    path = os.environ.get("RDN_PARITY_REPORT")
    s = err_stats(gpu, ref)
    s.update(test=test, tensor=tensor, elements=int(np.asarray(as64(ref)).size),
             beyond_plain_bound=excess_count(gpu, ref),
             stored_bf16=bool(isinstance(gpu, torch.Tensor) and gpu.dtype == torch.bfloat16),
             **extra)
    if path:
        with open(path, "a") as f:
            f.write(json.dumps(s) + "\n")
    return s
