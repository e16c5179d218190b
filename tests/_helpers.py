"""Shared helpers for the GPU parity tests (comparison rules and transfers).

Tolerances (fp32 accumulation of the CUDA path vs the fp64 oracle):
  * integer / index outputs and max reductions: bit-exact;
  * sum, mean, softmax: per element |gpu - oracle| <= TOL * scale, where
    scale is the oracle's sum of absolute terms (sum |w * x|, divided by the
    count for mean, sum alpha |x| for softmax).  TOL is 1e-5 for fp32
    features and 1e-2 for bf16 storage (the oracle reads the same bf16
    values, so the bf16 bound is loose by design).
"""
import numpy as np
import torch

TOL_F32 = 1e-5
TOL_BF16 = 1e-2


def dev(a: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def features(wl, dtype: str) -> torch.Tensor:
    if dtype == "bf16":
        bits = wl.x_bf16
        if bits is None:
            from paper_2101_11552_gb300.graphgen import bf16_bits_rne
            bits = bf16_bits_rne(wl.x)
        return dev(bits.view(np.int16)).view(torch.bfloat16)
    return dev(wl.x)


def host_features(wl, dtype: str) -> np.ndarray:
    """What the oracle reads: fp32 values, or the bf16 bit patterns."""
    if dtype == "bf16":
        if wl.x_bf16 is not None:
            return wl.x_bf16
        from paper_2101_11552_gb300.graphgen import bf16_bits_rne
        return bf16_bits_rne(wl.x)
    return wl.x


def assert_scaled_close(gpu: np.ndarray, ref: np.ndarray, scale: np.ndarray, tol: float,
                        what: str = ""):
    gpu = np.asarray(gpu, dtype=np.float64)
    diff = np.abs(gpu - ref)
    bound = tol * scale
    bad = diff > bound
    if bad.any():
        idx = np.argwhere(bad)[:5]
        worst = float(np.max(diff / np.maximum(scale, 1e-300)))
        raise AssertionError(
            f"{what}: {int(bad.sum())} of {bad.size} elements outside tol {tol} "
            f"(worst scaled error {worst:.3e}); first at {idx.tolist()}: "
            f"gpu={gpu[tuple(idx[0])]!r} oracle={ref[tuple(idx[0])]!r} scale={scale[tuple(idx[0])]!r}")


def alpha_scale(alpha_ref: np.ndarray) -> np.ndarray:
    """Error scale for attention weights: alpha itself plus an absolute floor
    of 1e-2 (so the bound is 1e-5 * alpha + 1e-7 at TOL_F32).  A weight
    exp(l - m) / den carries the fp32 rounding of its logit l as a relative
    error of about |l| * 2^-24 * (a few); with |l| ~ 30 that reaches ~1e-5 for
    weights far below anything that moves the output (1e-15 in practice),
    while the output itself is held to the full relative bound."""
    return np.asarray(alpha_ref) + 1e-2


def max_scaled_error(gpu, ref, scale) -> float:
    gpu = np.asarray(gpu, dtype=np.float64)
    s = np.where(scale > 0, scale, 1.0)
    return float(np.max(np.abs(gpu - ref) / s)) if gpu.size else 0.0


def assert_exact_f32(gpu: np.ndarray, ref_f64: np.ndarray, what: str = ""):
    """Max reductions: the fp32 result equals the oracle's exact value rounded to fp32."""
    want = ref_f64.astype(np.float32)
    got = np.asarray(gpu, dtype=np.float32)
    if not np.array_equal(got, want):     # -0.0 == +0.0 here, as intended
        bad = np.argwhere(got != want)[:5]
        raise AssertionError(f"{what}: {int((got != want).sum())} mismatches, first {bad.tolist()}: "
                             f"gpu={got[tuple(bad[0])]!r} oracle={want[tuple(bad[0])]!r}")
