"""Small numeric helpers for the tests (comparison metrics only)."""
import numpy as np


def rel_l2(a, b) -> float:
    """||a - b||_2 / ||b||_2 in float64 (0 when both are zero)."""
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    den = np.linalg.norm(b.ravel())
    num = np.linalg.norm((a - b).ravel())
    if den == 0.0:
        return float(num)
    return float(num / den)


def max_abs(a, b) -> float:
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    return float(np.max(np.abs(a - b))) if a.size else 0.0


def sigmoid_gap(r_full: np.ndarray, k: int) -> float:
    """Smallest gap between the k-th and (k+1)-th largest score over all rows."""
    flat = r_full.reshape(-1, r_full.shape[-1])
    if k >= flat.shape[1]:
        return float("inf")
    s = -np.sort(-flat, axis=1)
    return float(np.min(s[:, k - 1] - s[:, k]))
