"""CPU oracle for what a search does with the surrogate's 8-bin forecast.

TEST INFRASTRUCTURE ONLY (like ``oracle.model``).  Plain numpy, float64.

* Speedup bins and representatives: Table ``tab:speedup-bins`` (App. "Prompts"):
  bin 1 S <= 0.25, 2 (0.25, 0.5], 3 (0.5, 0.71], 4 (0.71, 1.0], 5 (1.0, 1.41],
  6 (1.41, 2.0], 7 (2.0, 4.0], 8 S > 4.0; interior representatives
  m_2..m_7 = 0.35, 0.59, 0.84, 1.19, 1.68, 2.83; the open bins' m_1 and m_8
  are empirical means the paper does not print, so they are parameters here.
* Expected speedup S_hat_i = sum_b p_ib m_b and speedup recovered over the
  budgets C = {1, 5, 10, 25, 50} % (Sec. 3.1).
* Expected calibration error over ten confidence buckets and forecast error
  (Sec. 3.1); Brier and CRPS scores (Sec. 2.2).
* Discovery moments (Sec. 3.6): s = Pr[g >= x] from the forecast distribution
  and y_hat = 1[s >= tau].

Readings where the paper is silent:
* Top_c takes ceil(c * n / 100) candidates, at least one, ranked by S_hat
  (ties: lower index first).
* ECE buckets are ten equal-width confidence intervals (0, 0.1], ..., (0.9, 1.0]
  (a confidence of exactly 0 goes to the first bucket).
* Pr[g >= x] sums the mass of the bins that lie entirely at or above x, i.e.
  whose lower edge is >= x (the bin edges do not fall on 1.25 or 1.5).
"""
from __future__ import annotations

import math

import numpy as np

UPPER_EDGES = (0.25, 0.5, 0.71, 1.0, 1.41, 2.0, 4.0)          # upper edges of bins 1..7
LOWER_EDGES = (0.0, 0.25, 0.5, 0.71, 1.0, 1.41, 2.0, 4.0)     # lower edges of bins 1..8
INTERIOR_REPRESENTATIVES = (0.35, 0.59, 0.84, 1.19, 1.68, 2.83)  # m_2 .. m_7
BUDGETS = (1, 5, 10, 25, 50)


def speedup_bin(S: float) -> int:
    """Bin 1..8 of a measured speedup (upper edges inclusive)."""
    for b, edge in enumerate(UPPER_EDGES, start=1):
        if S <= edge:
            return b
    return 8


def representatives(m1: float, m8: float) -> np.ndarray:
    return np.array([m1, *INTERIOR_REPRESENTATIVES, m8], dtype=np.float64)


def expected_speedup(p: np.ndarray, m: np.ndarray) -> np.ndarray:
    """S_hat = sum_b p_b m_b for each row of p ([n, 8])."""
    return np.asarray(p, dtype=np.float64) @ np.asarray(m, dtype=np.float64)


def ranking(s_hat: np.ndarray) -> np.ndarray:
    """Indices by decreasing S_hat, lower index first among equals."""
    s_hat = np.asarray(s_hat, dtype=np.float64)
    return np.array(sorted(range(len(s_hat)), key=lambda i: (-s_hat[i], i)), dtype=np.int64)


def top_count(n: int, c: float) -> int:
    return max(1, math.ceil(c * n / 100.0))


def recovered(s_hat: np.ndarray, S: np.ndarray, budgets=BUDGETS) -> float:
    """100/|C| * sum_c max_{i in Top_c} S_i / max_i S_i."""
    S = np.asarray(S, dtype=np.float64)
    order = ranking(s_hat)
    best = S.max()
    return 100.0 / len(budgets) * sum(S[order[:top_count(len(S), c)]].max() / best for c in budgets)


def ece(conf: np.ndarray, correct: np.ndarray, n_buckets: int = 10) -> float:
    """sum_m |B_m|/n |acc(B_m) - conf(B_m)| over equal-width confidence buckets."""
    conf = np.asarray(conf, dtype=np.float64)
    correct = np.asarray(correct, dtype=np.float64)
    n = len(conf)
    bucket = np.clip(np.ceil(conf * n_buckets).astype(int) - 1, 0, n_buckets - 1)
    total = 0.0
    for m in range(n_buckets):
        sel = bucket == m
        if sel.any():
            total += sel.sum() / n * abs(correct[sel].mean() - conf[sel].mean())
    return total


def forecast_error(pred_bin: np.ndarray, S: np.ndarray, m: np.ndarray) -> float:
    """mean |m_{y_hat} - S| (bins numbered 1..8)."""
    m = np.asarray(m, dtype=np.float64)
    return float(np.mean(np.abs(m[np.asarray(pred_bin) - 1] - np.asarray(S, dtype=np.float64))))


def brier(p: np.ndarray, y: int) -> float:
    """1/2 sum_b (p_b - 1[b = y])^2, y in 1..8."""
    onehot = np.zeros(8)
    onehot[y - 1] = 1.0
    return 0.5 * float(np.sum((np.asarray(p, dtype=np.float64) - onehot) ** 2))


def crps(p: np.ndarray, y: int) -> float:
    """1/7 sum_{k=1..7} (F_k - 1[y <= k])^2 with F_k the cumulative forecast."""
    F = np.cumsum(np.asarray(p, dtype=np.float64))[:7]
    target = np.array([1.0 if y <= k else 0.0 for k in range(1, 8)])
    return float(np.sum((F - target) ** 2) / 7.0)


def discovery_score(p: np.ndarray, x: float) -> np.ndarray:
    """s = Pr[g >= x]: the forecast mass of the bins whose lower edge is >= x."""
    mask = np.array([lo >= x for lo in LOWER_EDGES], dtype=np.float64)
    return np.asarray(p, dtype=np.float64) @ mask


def discovery_predict(s: np.ndarray, tau: float) -> np.ndarray:
    """y_hat = 1[s >= tau]."""
    return (np.asarray(s) >= tau).astype(np.uint8)
