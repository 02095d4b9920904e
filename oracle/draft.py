"""Base draft policy D: reuse and the order-K Taylor draft (Eq. 2), float64.

What is forecast.  The draft of block l at step t is h^d = D(u) (Eq. 3), a
function of the incoming state u.  The forecast quantity is the block's
residual increment R_{s,l} = h^f_{s,l} - u_{s,l} stored at exact refreshes s,
and the draft is h^d = u + forecast.  With K = 0 this is reuse of the last
refreshed increment.

Eq. 2 writes the order-K draft as sum_k (t - s)^k / k! * Delta^(k)_s with the
derivative estimates Delta^(k) taken from finite differences at exact
refreshes.  Two estimators are provided:

* ``"interp"`` (default): Delta^(k) is the k-th derivative at s_0 of the
  polynomial that interpolates the last K_eff + 1 refreshed increments
  (Newton divided differences).  It is exact on increments that are
  polynomials of degree <= K_eff in the step index.
* ``"recursive"``: Delta^(0)_{s_j} = R_{s_j} and
  Delta^(k)_{s_j} = (Delta^(k-1)_{s_j} - Delta^(k-1)_{s_{j+1}}) / (s_j - s_{j+1}),
  each level divided by the spacing between the two refreshes it joins.
  Equal to ``"interp"`` for K <= 1; for K >= 2 it is not exact on
  quadratics.

The oracle forms the Delta^(k) tensors explicitly and sums the Taylor series
(Eq. 2 as written).  It never forms per-refresh scalar weights, so the GPU
path's weight form is checked against an independent route.

Test infrastructure only.
"""

import math

import numpy as np


def _poly_in_tau(nodes_minus_s0):
    """Coefficients (ascending powers of tau = t - s_0) of prod_j (tau - a_j)."""
    coef = np.array([1.0])
    for a in nodes_minus_s0:
        nxt = np.zeros(len(coef) + 1)
        nxt[1:] += coef          # tau * p(tau)
        nxt[:-1] -= a * coef     # -a * p(tau)
        coef = nxt
    return coef


def divided_differences(s, R):
    """Newton divided differences [s_0], [s_0, s_1], ... of tensors R at nodes s."""
    n = len(s)
    table = [np.asarray(r, dtype=np.float64) for r in R]
    out = [table[0]]
    for m in range(1, n):
        table = [(table[j] - table[j + 1]) / (s[j] - s[j + m]) for j in range(n - m)]
        out.append(table[0])
    return out


def derivative_estimates(s, R, variant="interp"):
    """Delta^(k) at s_0 for k = 0 .. len(s) - 1 (Eq. 2's finite differences).

    ``s`` lists refresh steps newest first, ``R`` the matching increments.
    """
    K = len(s) - 1
    if variant == "recursive":
        level = [np.asarray(r, dtype=np.float64) for r in R]
        D = [level[0]]
        for k in range(1, K + 1):
            level = [(level[j] - level[j + 1]) / (s[j] - s[j + 1]) for j in range(len(level) - 1)]
            D.append(level[0])
        return D
    if variant != "interp":
        raise ValueError("unknown Taylor variant %r" % variant)
    dd = divided_differences(s, R)
    # Newton basis polynomial m is prod_{j<m} (t - s_j); in tau = t - s_0 its
    # nodes sit at s_j - s_0.  Its coefficient of tau^k times k! is its k-th
    # derivative at s_0.
    D = [np.zeros_like(dd[0]) for _ in range(K + 1)]
    for m in range(K + 1):
        coef = _poly_in_tau([s[j] - s[0] for j in range(m)])
        for k in range(len(coef)):
            if coef[k] != 0.0:
                D[k] = D[k] + math.factorial(k) * coef[k] * dd[m]
    return D


def taylor_forecast(t, s, R, variant="interp"):
    """sum_k (t - s_0)^k / k! * Delta^(k)_{s_0}   (Eq. 2)."""
    D = derivative_estimates(s, R, variant)
    out = np.zeros_like(D[0])
    for k, Dk in enumerate(D):
        out = out + (t - s[0]) ** k / math.factorial(k) * Dk
    return out


def draft(u, history, t, K, variant="interp"):
    """h^d = u + forecast of the block increment from its refresh history.

    ``history`` is a list of (refresh_step, increment) newest first; the
    effective order is min(K, len(history) - 1) (fewer refreshes than K + 1
    lower the order; one refresh gives reuse).
    """
    k_eff = min(K, len(history) - 1)
    s = [history[j][0] for j in range(k_eff + 1)]
    R = [history[j][1] for j in range(k_eff + 1)]
    return np.asarray(u, dtype=np.float64) + taylor_forecast(t, s, R, variant)
