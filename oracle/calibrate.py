"""Offline key-channel selection of DAMP, in float64 numpy.  Test infrastructure only.

Follows Sec. 5.1 (Eq. budgeted_allocation, error_energy, persistence,
budgeted_selection), App. A.2 (Eq. domain_balanced_calibration,
empirical_error_energy, empirical_persistence) and Algorithm 1 (App. A.4):

  E_u    = E_cal || [Q_lo(S)]_{u:} - S_{u:} ||_2^2          quantization-error energy
  a_eff  = exp(E_cal[log a_{t,u}])                          geometric-mean retention
  P_u    = 1 / max(1 - a_eff_u^2, tau),  tau = 1e-4         capped persistence
  C_u    = E_u * P_u                                        accumulated-error risk
  H      = TopK_{K_hi}(C)                                   protected channels
  pi     = stable partition placing H before its complement

Readings where the paper is silent: TopK breaks ties in favour of the lower
channel index; the stable partition keeps ascending channel order inside H and
inside its complement; E_cal over a single synthetic domain is the plain mean.
"""
from __future__ import annotations

import numpy as np

from . import core

TAU = 1e-4


def domain_balanced_mean(values: np.ndarray, domains=None) -> np.ndarray:
    """E_cal[f] = (1/|D|) sum_d (1/|Omega_d|) sum_{x in Omega_d} f(x) over axis 0.

    `domains` is a list of index arrays (one per domain) into axis 0; None means
    one domain holding every sample (the plain mean).
    """
    values = np.asarray(values, dtype=np.float64)
    if domains is None:
        return values.mean(axis=0)
    return np.mean([values[np.asarray(idx)].mean(axis=0) for idx in domains], axis=0)


def error_energy_samples(states: np.ndarray, fmt: int) -> np.ndarray:
    """Per-sample, per-key-channel squared reconstruction error ||Q_lo(S)_u - S_u||^2.

    states: float32 [n_samples, d_k, d_v] natural-order states of one head.
    Returns float64 [n_samples, d_k].
    """
    rec = core.qdq_rows(states, fmt).astype(np.float64)
    return ((rec - states.astype(np.float64)) ** 2).sum(axis=-1)


def error_energy(states: np.ndarray, fmt: int, domains=None) -> np.ndarray:
    """E_u (Eq. empirical_error_energy) over calibration state samples of one head."""
    return domain_balanced_mean(error_energy_samples(states, fmt), domains)


def effective_decay(log_a: np.ndarray, domains=None) -> np.ndarray:
    """a_eff = exp(E_cal[log a]) over axis 0 (the calibration steps)."""
    return np.exp(domain_balanced_mean(log_a, domains))


def persistence(a_eff, tau: float = TAU) -> np.ndarray:
    """P = min(sum_j a_eff^{2j}, 1/tau) = 1 / max(1 - a_eff^2, tau) (Eq. persistence)."""
    a_eff = np.asarray(a_eff, dtype=np.float64)
    return 1.0 / np.maximum(1.0 - a_eff ** 2, tau)


def topk(scores, k: int) -> np.ndarray:
    """Indices of the k largest scores; equal scores prefer the lower index."""
    scores = np.asarray(scores, dtype=np.float64)
    order = sorted(range(scores.size), key=lambda u: (-scores[u], u))
    return np.array(sorted(order[:k]), dtype=np.int64)


def stable_partition(protected, d_k: int) -> np.ndarray:
    """pi: the protected channels first, then the rest, each in ascending channel order."""
    mark = np.zeros(d_k, dtype=bool)
    mark[np.asarray(protected, dtype=np.int64)] = True
    first = [u for u in range(d_k) if mark[u]]
    rest = [u for u in range(d_k) if not mark[u]]
    return np.array(first + rest, dtype=np.uint8)


def select_layout(E, P, k_hi: int):
    """Algorithm 1 for one (layer, head): C = E * P, H = TopK(C), pi = stable partition."""
    C = np.asarray(E, dtype=np.float64) * np.asarray(P, dtype=np.float64)
    H = topk(C, k_hi)
    return H, stable_partition(H, C.size)


def bits_budgeted(k_hi: int, d_k: int, b_hi: float, b_lo: float) -> float:
    """b(K_hi) = b_lo + (K_hi / d_k)(b_hi - b_lo)  (Eq. budgeted_allocation)."""
    return b_lo + (k_hi / d_k) * (b_hi - b_lo)
