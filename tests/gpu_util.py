"""Helpers for the GPU parity tests (tolerances from the stated parity bar)."""
import numpy as np

ENTROPY_ATOL = 1e-3      # nats, absolute
IMPORTANCE_RTOL = 1e-2   # relative, element by element
POOLED_RTOL = 2e-3       # max-abs error / max-abs value of the oracle vector
PRED_ATOL = 1.0          # tokens


def assert_entropy(gpu, ref):
    gpu, ref = np.asarray(gpu, np.float64), np.asarray(ref, np.float64)
    err = np.max(np.abs(gpu - ref)) if ref.size else 0.0
    assert err <= ENTROPY_ATOL, f"entropy max abs err {err:.3e}"
    return err


def assert_importance(gpu, ref):
    gpu, ref = np.asarray(gpu, np.float64), np.asarray(ref, np.float64)
    rel = np.abs(gpu - ref) / np.maximum(np.abs(ref), 1e-30)
    bad = rel > IMPORTANCE_RTOL
    assert not bad.any(), f"importance rel err {rel.max():.3e} at {np.nonzero(bad)[0][:8]}"
    return rel.max() if rel.size else 0.0


def assert_pooled(gpu, ref):
    gpu, ref = np.asarray(gpu, np.float64), np.asarray(ref, np.float64)
    for b in range(ref.shape[0]):
        scale = np.max(np.abs(ref[b]))
        err = np.max(np.abs(gpu[b] - ref[b]))
        assert err <= POOLED_RTOL * scale + 1e-30, f"pooled row {b}: err {err:.3e} scale {scale:.3e}"


def assert_pred(gpu, ref):
    err = np.max(np.abs(np.asarray(gpu, np.float64) - np.asarray(ref, np.float64)))
    assert err <= PRED_ATOL, f"predicted length err {err:.3f}"
