"""Helpers shared by the GPU parity tests (no method arithmetic here)."""
import numpy as np
import torch


def cuda(a, dtype=None):
    t = torch.as_tensor(np.ascontiguousarray(a))
    if dtype is not None:
        t = t.to(dtype)
    return t.cuda()


def rel_err_floor(got, want, floor):
    got = np.asarray(got, np.float64)
    want = np.asarray(want, np.float64)
    return np.abs(got - want) / np.maximum(np.abs(want), floor)


def rel_l2(got, want):
    got = np.asarray(got, np.float64)
    want = np.asarray(want, np.float64)
    den = np.linalg.norm(want)
    return float(np.linalg.norm(got - want) / (den if den > 0 else 1.0))


def near_bound(logp, old, eps_low, eps_high, tol=1e-6):
    """Tokens whose ratio lies within tol of a clip bound (mask parity excludes them)."""
    r = np.exp(np.asarray(logp, np.float64) - np.asarray(old, np.float64))
    with np.errstate(invalid="ignore"):
        return (np.abs(r - (1.0 - eps_low)) <= tol) | (np.abs(r - (1.0 + eps_high)) <= tol)
