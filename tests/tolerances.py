"""Comparison rules of the parity tests (GPU path vs oracle), one per output kind.

bf16 perturbed weights: at most 1 bf16 ulp of the largest operand of the fma
    (theta, sigma eps or the exact result) apart -- under cancellation the result's own
    ulp can be far smaller than any fp32 evaluation error -- and bit-exact in >= 99.9%.
fp32 perturbed weights: |d| <= 1e-6 * max(|w|, |theta|, |sigma eps|) -- relative to the
    largest operand of the single fma, so cancellation cannot make it unreachable.
fp32 updated master: |d| <= 1e-6 * max(|theta+|, |c| sum_j |w_j eps_j|) -- relative to
    the magnitude of the terms summed (the error of any fp32 evaluation scales with it).
normals: |d| <= 2^-20 * max(1, |eps|).
shaped fitness: |d| <= 1e-6 * |f| + 2^-40.
"""
import numpy as np


def bf16_order(bits):
    b = np.asarray(bits, dtype=np.int64) & 0xFFFF
    mag = b & 0x7FFF
    return np.where(b & 0x8000, -mag, mag)


def bf16_ulp_diff(a_bits, b_bits):
    return np.abs(bf16_order(a_bits) - bf16_order(b_bits))


def bf16_value(bits):
    b = np.asarray(bits, dtype=np.uint32) << 16
    return b.view(np.float32).astype(np.float64)


def bf16_ulp(v):
    """Spacing of bf16 values at magnitude v (8 significant bits; subnormal floor 2^-133)."""
    v = np.maximum(np.abs(np.asarray(v, dtype=np.float64)), 2.0**-126)
    return np.exp2(np.floor(np.log2(v)) - 7)


def assert_bf16_close(got_bits, ref_bits, scale=None, min_exact=0.999):
    """scale: magnitude of the largest operand per element (None: the result itself)."""
    d = bf16_ulp_diff(got_bits, ref_bits)
    exact = float(np.mean(d == 0)) if d.size else 1.0
    if d.size:
        ref = bf16_value(ref_bits)
        mag = np.abs(ref) if scale is None else np.maximum(np.abs(ref), np.abs(scale))
        err = np.abs(bf16_value(got_bits) - ref)
        assert np.all(err <= bf16_ulp(mag)), f"bf16 differs by {d.max()} ulp of the result"
    assert exact >= min_exact, f"only {exact:.6f} bit-exact"
    return exact


def assert_perturb_fp32_close(got, ref_exact, theta, sigma_eps):
    tol = 1e-6 * np.maximum.reduce([np.abs(ref_exact), np.abs(theta), np.abs(sigma_eps)])
    err = np.abs(got.astype(np.float64) - ref_exact)
    assert np.all(err <= tol), f"max err/tol {np.max(err / np.maximum(tol, 1e-300)):.3g}"


def assert_update_close(got, ref_exact, scale):
    tol = 1e-6 * np.maximum(np.abs(ref_exact), scale)
    err = np.abs(got.astype(np.float64) - ref_exact)
    ratio = err / np.maximum(tol, 1e-300)
    assert np.all(err <= tol), f"max err/tol {ratio.max():.3g}"
    return float(ratio.max()) if ratio.size else 0.0


def assert_normals_close(got, ref):
    err = np.abs(got.astype(np.float64) - ref)
    tol = 2.0**-20 * np.maximum(1.0, np.abs(ref))
    assert np.all(err <= tol), f"max err/tol {np.max(err / tol):.3g}"


def assert_fitness_close(got, ref):
    err = np.abs(got.astype(np.float64) - ref.astype(np.float64))
    assert np.all(err <= 1e-6 * np.abs(ref) + 2.0**-40), f"max err {err.max():.3g}"
