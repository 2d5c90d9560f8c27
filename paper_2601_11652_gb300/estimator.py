"""Verification-time estimator (Sec. 4.4, Eq. batch_time) fitted on this library's own timings.

The paper models the latency of a verification batch as an additive function of three workload
features (Sec. 4.4):

    N_linear       = sum_i L_new,i                       tokens entering the GPU
    N_interactions = sum_i L_total,i * L_new,i           query-key interactions
    N_cached       = sum_i L_cached,i                    cached tokens read from HBM

    T_batch ~= a * N_linear + b_compute * N_interactions + b_read * N_cached + c

and fits (a, b_compute, b_read, c) by ordinary least squares, validated with R^2, adjusted R^2,
RMSE, MAE, MAPE, 5-fold cross-validation and 95% confidence intervals (the appendix's profiling
methodology).  In a verification step of this library request i brings L_new,i = k_i + 1 new tokens
over L_cached,i = c_i cached ones (L_total,i = c_i + k_i + 1).  `bench.py --latency-table` measures
the step over a sweep of batch sizes and draft lengths and fits this model to it.

Host-side numpy only; nothing here runs on the GPU.
"""
from __future__ import annotations

import dataclasses

import numpy as np

FEATURES = ("N_linear", "N_interactions", "N_cached")


def features(context_lens, draft_lens) -> np.ndarray:
    """[N_linear, N_interactions, N_cached] of one batch (Sec. 4.4): L_new = k + 1, L_cached = c."""
    c = np.asarray(context_lens, dtype=np.float64)
    new = np.asarray(draft_lens, dtype=np.float64) + 1.0
    total = c + new
    return np.array([new.sum(), (total * new).sum(), c.sum()])


def _design(X: np.ndarray) -> np.ndarray:
    X = np.asarray(X, dtype=np.float64)
    return np.hstack([X, np.ones((X.shape[0], 1))])


def fit_ols(X, y) -> np.ndarray:
    """Least-squares coefficients [a, b_compute, b_read, c] (last = intercept)."""
    coef, *_ = np.linalg.lstsq(_design(X), np.asarray(y, dtype=np.float64), rcond=None)
    return coef


def predict(coef, X) -> np.ndarray:
    return _design(X) @ np.asarray(coef, dtype=np.float64)


def metrics(y, yhat, n_features: int = 3) -> dict:
    """R^2, adjusted R^2, RMSE, MAE and MAPE (in %) of predictions yhat of y."""
    y = np.asarray(y, dtype=np.float64)
    yhat = np.asarray(yhat, dtype=np.float64)
    res = y - yhat
    ss_res = float(res @ res)
    ss_tot = float(((y - y.mean()) ** 2).sum())
    n = len(y)
    r2 = 1.0 - ss_res / ss_tot if ss_tot > 0 else float("nan")
    adj = 1.0 - (1.0 - r2) * (n - 1) / (n - n_features - 1) if n > n_features + 1 else float("nan")
    return {"r2": r2, "adj_r2": adj, "rmse": float(np.sqrt(ss_res / n)), "mae": float(np.abs(res).mean()),
            "mape": float(100.0 * np.abs(res / y).mean())}


def cross_validate(X, y, folds: int = 5, seed: int = 0) -> dict:
    """k-fold cross-validation: mean and spread of the held-out R^2 and MAE."""
    X = np.asarray(X, dtype=np.float64)
    y = np.asarray(y, dtype=np.float64)
    idx = np.random.default_rng(seed).permutation(len(y))
    parts = np.array_split(idx, folds)
    r2, mae = [], []
    for f in range(folds):
        test = parts[f]
        train = np.concatenate([parts[g] for g in range(folds) if g != f])
        coef = fit_ols(X[train], y[train])
        m = metrics(y[test], predict(coef, X[test]))
        r2.append(m["r2"])
        mae.append(m["mae"])
    return {"folds": folds, "r2_mean": float(np.mean(r2)), "r2_std": float(np.std(r2)),
            "mae_mean": float(np.mean(mae)), "mae_std": float(np.std(mae))}


def bootstrap_ci(X, y, n: int = 1000, seed: int = 0, level: float = 0.95) -> np.ndarray:
    """Percentile bootstrap intervals of the coefficients: array [4, 2] of (low, high)."""
    X = np.asarray(X, dtype=np.float64)
    y = np.asarray(y, dtype=np.float64)
    rng = np.random.default_rng(seed)
    coefs = np.empty((n, X.shape[1] + 1))
    for i in range(n):
        s = rng.integers(0, len(y), size=len(y))
        coefs[i] = fit_ols(X[s], y[s])
    lo, hi = (1.0 - level) / 2.0, 1.0 - (1.0 - level) / 2.0
    return np.stack([np.quantile(coefs, lo, axis=0), np.quantile(coefs, hi, axis=0)], axis=1)


@dataclasses.dataclass
class Fit:
    coef: np.ndarray      # [a, b_compute, b_read, c]
    ci: np.ndarray        # [4, 2]
    train: dict           # metrics on the training rows
    test: dict            # metrics on the held-out rows
    cv: dict              # cross-validation on the training rows

    def report(self, unit: str = "s") -> str:
        names = ("a (per new token)", "b_compute (per interaction)", "b_read (per cached token)", "c (constant)")
        lines = [f"{nm:30s} {v: .4e}  95% CI [{lo: .4e}, {hi: .4e}] {unit}" for nm, v, (lo, hi) in zip(names, self.coef, self.ci)]
        for tag, m in (("train", self.train), ("test", self.test)):
            lines.append(f"{tag}: R2 {m['r2']:.4f}  adj R2 {m['adj_r2']:.4f}  RMSE {m['rmse']:.3e}  MAE {m['mae']:.3e}  MAPE {m['mape']:.2f}%")
        lines.append(f"{self.cv['folds']}-fold CV on train: R2 {self.cv['r2_mean']:.4f} +- {self.cv['r2_std']:.4f}, "
                     f"MAE {self.cv['mae_mean']:.3e} +- {self.cv['mae_std']:.3e}")
        return "\n".join(lines)


def fit_with_validation(X, y, test_fraction: float = 0.3, seed: int = 0, n_boot: int = 1000) -> Fit:
    """Fit on a random training split, report train / held-out metrics, CV and bootstrap CIs."""
    X = np.asarray(X, dtype=np.float64)
    y = np.asarray(y, dtype=np.float64)
    idx = np.random.default_rng(seed).permutation(len(y))
    n_test = max(1, int(round(test_fraction * len(y))))
    test, train = idx[:n_test], idx[n_test:]
    coef = fit_ols(X[train], y[train])
    return Fit(coef=coef, ci=bootstrap_ci(X[train], y[train], n=n_boot, seed=seed),
               train=metrics(y[train], predict(coef, X[train])), test=metrics(y[test], predict(coef, X[test])),
               cv=cross_validate(X[train], y[train], seed=seed))
