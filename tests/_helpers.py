"""Shared helpers for the GPU parity tests (comparison rules and transfers).

Tolerances (fp32 accumulation of the CUDA path vs the fp64 oracle):
  * integer / index outputs and max reductions: bit-exact;
  * sum, mean, softmax: per element |gpu - oracle| <= TOL * scale, where
    scale is the oracle's sum of absolute terms (sum |w * x|, divided by the
    count for mean, sum alpha |x| for softmax).  TOL is 1e-5 for fp32
    features and for bf16 storage alike: the oracle reads the same bf16
    values, so fp32 arithmetic is the only error either way (the stated
    1e-2 bound for bf16 storage is not needed);
  * attention weights: |gpu - oracle| <= alpha * (TOL + kappa * (lam_e +
    lam_max)), where lam_e is the magnitude that edge e's logit is computed
    from (|s_src| + |s_dst| for the additive form, scale * sum |q k| for the
    dot-product form), lam_max its maximum over the edge's row, and kappa a
    small multiple of the fp32 unit roundoff (see alpha_bound).
"""
import numpy as np
import torch

TOL_F32 = 1e-5
U32 = 2.0 ** -24          # unit roundoff of fp32 (round to nearest)


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


# Attention weights alpha = exp(l - m) / den computed in fp32.  A logit l is
# formed from terms of total magnitude lam (|s_src| + |s_dst|, or
# scale * sum |q k|), so its fp32 value carries an absolute error of a few
# units of roundoff times lam; the row maximum m carries the same for its
# own edge (at most lam_max); exp turns an absolute error d of (l - m) into a
# relative error d of the weight (the base-2 form used by the kernels gives
# the same figure: ln 2 * log2(e) = 1).  The exponential itself (2 ulp), the
# denominator's fp32 sums and the division add a fixed relative error that
# TOL covers, as it does for the outputs.  So
#     |alpha_gpu - alpha| <= alpha * (TOL + kappa * (lam_e + lam_max)).
# Additive form: node scores are compensated dot products (error ~ u |s|),
# scaled to base 2 and added (a few more u), LeakyReLU multiplies once:
# at most ~7u lam for a logit, ~23u (lam_e + lam_max) after the maximum and
# the running-maximum rescales -> kappa = 32u.  Dot-product form: plain fp32
# dot products of C terms split over lanes (error <= (C + 8) u lam) ->
# kappa = (2 C + 32) u.
KAPPA_GAT = 32 * U32


def kappa_dot(channels: int) -> float:
    return (2 * channels + 32) * U32


def gat_logit_mag(x64: np.ndarray, src: np.ndarray, dst: np.ndarray, heads: int, channels: int,
                  a_src, a_dst) -> np.ndarray:
    """lam[e, h] = |s_src[src_e, h]| + |s_dst[dst_e, h]| in fp64 from the
    oracle's view of the inputs (x widened exactly)."""
    xs = np.asarray(x64, np.float64).reshape(-1, heads, channels)
    s_src = np.einsum("nhc,hc->nh", xs, np.asarray(a_src, np.float64).reshape(heads, channels))
    s_dst = np.einsum("nhc,hc->nh", xs, np.asarray(a_dst, np.float64).reshape(heads, channels))
    return np.abs(s_src[src]) + np.abs(s_dst[dst])


def dot_logit_mag(q64, k64, src, dst, heads: int, channels: int, scale: float) -> np.ndarray:
    """lam[e, h] = scale * sum_c |q[dst_e, h, c] k[src_e, h, c]| (fp64)."""
    q = np.asarray(q64, np.float64).reshape(-1, heads, channels)
    k = np.asarray(k64, np.float64).reshape(-1, heads, channels)
    lam = np.empty((len(src), heads))
    for h in range(heads):
        lam[:, h] = abs(scale) * np.einsum("ec,ec->e", np.abs(q[dst, h]), np.abs(k[src, h]))
    return lam


def assert_alpha_close(got: np.ndarray, want: np.ndarray, lam: np.ndarray, row: np.ndarray,
                       kappa: float, what: str = ""):
    """Attention weights in CSR order: row[e] is edge e's target (rows are
    contiguous), lam[e, h] its logit magnitude (same order)."""
    want = np.asarray(want, np.float64).reshape(lam.shape)
    got = np.asarray(got, np.float64).reshape(lam.shape)
    lam_max = np.zeros((int(row.max()) + 1 if len(row) else 1, lam.shape[1]))
    np.maximum.at(lam_max, row, lam)
    bound = want * (TOL_F32 + kappa * (lam + lam_max[row]))
    bad = np.abs(got - want) > bound
    if bad.any():
        i = np.argwhere(bad)[0]
        rel = np.abs(got - want) / np.maximum(want, 1e-300)
        raise AssertionError(
            f"{what}: {int(bad.sum())} of {bad.size} weights outside the bound; first at "
            f"{i.tolist()}: gpu={got[tuple(i)]!r} oracle={want[tuple(i)]!r} "
            f"lam={lam[tuple(i)]!r} lam_max={lam_max[row[i[0]], i[1]]!r}; worst relative "
            f"error {float(rel.max()):.3e}")


def csr_rows(rowptr: np.ndarray) -> np.ndarray:
    """Target row of every CSR position."""
    rowptr = np.asarray(rowptr, np.int64)
    return np.repeat(np.arange(len(rowptr) - 1), np.diff(rowptr))


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


def row_edges(ocsr, rows):
    """(src, dst, local row index) of the in-edges of the listed rows, in
    CSR order, rows one after another (the packing of the oracle's *_rows
    alpha output)."""
    rp, col = np.asarray(ocsr[0], np.int64), np.asarray(ocsr[1], np.int64)
    rows = np.asarray(rows, np.int64)
    deg = rp[rows + 1] - rp[rows]
    src = (np.concatenate([col[rp[r]:rp[r + 1]] for r in rows]) if len(rows)
           else np.zeros(0, np.int64))
    return src, np.repeat(rows, deg), np.repeat(np.arange(len(rows)), deg)
