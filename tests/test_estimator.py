"""The verification-time estimator (Sec. 4.4): features, OLS fit and validation metrics (CPU)."""
import numpy as np

from paper_2601_11652_gb300 import estimator as est


def test_features_follow_the_definitions():
    # two requests: c = (100, 0), k = (3, 7): L_new = (4, 8), L_total = (104, 8)
    f = est.features([100, 0], [3, 7])
    assert f.tolist() == [12.0, 104 * 4 + 8 * 8, 100.0]


def _synthetic(n=200, noise=0.0, seed=1):
    rng = np.random.default_rng(seed)
    X = np.column_stack([rng.uniform(10, 5000, n), rng.uniform(1e4, 5e7, n), rng.uniform(100, 3e6, n)])
    coef = np.array([3.3e-5, 3.45e-8, 4.6e-6, 1.5e-2])
    y = X @ coef[:3] + coef[3]
    return X, y * (1.0 + noise * rng.standard_normal(n)), coef


def test_ols_recovers_exact_coefficients():
    X, y, coef = _synthetic()
    got = est.fit_ols(X, y)
    np.testing.assert_allclose(got, coef, rtol=1e-6)
    m = est.metrics(y, est.predict(got, X))
    assert m["r2"] > 1 - 1e-12 and m["mae"] < 1e-9 and m["mape"] < 1e-6


def test_ols_matches_normal_equations():
    X, y, _ = _synthetic(noise=0.02)
    A = np.hstack([X, np.ones((len(y), 1))])
    np.testing.assert_allclose(est.fit_ols(X, y), np.linalg.solve(A.T @ A, A.T @ y), rtol=1e-6)


def test_metrics_definitions():
    y = np.array([1.0, 2.0, 3.0, 4.0, 5.0, 6.0])
    yhat = np.array([1.5, 2.0, 2.5, 4.0, 5.5, 6.0])
    m = est.metrics(y, yhat)
    res = y - yhat
    assert np.isclose(m["rmse"], np.sqrt((res ** 2).mean()))
    assert np.isclose(m["mae"], np.abs(res).mean())
    assert np.isclose(m["mape"], 100 * np.abs(res / y).mean())
    r2 = 1 - (res ** 2).sum() / ((y - y.mean()) ** 2).sum()
    assert np.isclose(m["r2"], r2)
    assert np.isclose(m["adj_r2"], 1 - (1 - r2) * 5 / 2)


def test_validation_with_noise_covers_the_truth():
    X, y, coef = _synthetic(noise=0.01, n=300)
    fit = est.fit_with_validation(X, y, seed=3, n_boot=300)
    assert fit.train["r2"] > 0.99 and fit.test["r2"] > 0.99
    assert fit.cv["folds"] == 5 and fit.cv["r2_mean"] > 0.99
    # the 95% bootstrap intervals of the slopes contain the generating values
    for j in range(3):
        assert fit.ci[j, 0] <= coef[j] <= fit.ci[j, 1], (j, fit.ci[j], coef[j])
    assert "b_read" in fit.report()
