"""Helpers shared by the GPU parity tests (no arithmetic of the method here)."""

import numpy as np
import torch

# Tolerances stated for the path: |dlogp| <= 2e-3, |dH| <= 2e-3, relative
# ratio error <= 1e-3, keep-mask exact outside a 1e-4 band around the
# threshold, relative gradient error <= 1e-2.
TOL_LOGP = 2e-3
TOL_ENT = 2e-3
TOL_RATIO = 1e-3
MASK_BAND = 1e-4
TOL_GRAD = 1e-2


def cuda(t):
    return t.to("cuda") if isinstance(t, torch.Tensor) else t


def np_(t):
    return t.detach().cpu().numpy()


def assert_close_abs(got, want, tol, what):
    got = np.asarray(got, dtype=np.float64)
    want = np.asarray(want, dtype=np.float64)
    assert got.shape == want.shape, (what, got.shape, want.shape)
    assert np.all(np.isfinite(got)), f"{what}: non-finite values"
    err = np.abs(got - want)
    i = int(np.argmax(err)) if err.size else 0
    assert err.size == 0 or err.max() <= tol, f"{what}: max |diff| {err.max():.3e} at {i} (tol {tol})"


def assert_close_rel(got, want, tol, what):
    got = np.asarray(got, dtype=np.float64)
    want = np.asarray(want, dtype=np.float64)
    err = np.abs(got - want) / np.maximum(np.abs(want), 1e-30)
    assert err.size == 0 or err.max() <= tol, f"{what}: max rel diff {err.max():.3e} (tol {tol})"


def assert_masks_match(got, want, stat, delta, band, what):
    """Masks equal except where the statistic is within `band` of the threshold."""
    got = np.asarray(got).astype(bool)
    want = np.asarray(want).astype(bool)
    near = np.abs(np.asarray(stat, dtype=np.float64) - delta) <= band
    bad = (got != want) & ~near
    assert not bad.any(), f"{what}: mask differs at {np.nonzero(bad)[0][:10]}"


def rel_fro(got, want):
    got = np.asarray(got, dtype=np.float64)
    want = np.asarray(want, dtype=np.float64)
    return np.linalg.norm(got - want) / max(np.linalg.norm(want), 1e-300)
