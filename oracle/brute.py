"""Quadratic-time definition of eq. 2, fp64, for tiny inputs.

ORACLE -- test infrastructure only; see oracle/__init__.py.

att_lin_quadratic is the first form of eq. 2 written out row by row: for every
position l, a weighted average of the values V_{l'} with l' <= l (inclusive
causal mask, Sec. 2.1), the weight of l' being g(K_{l'})^T g(Q_l).

Shapes: Q, K, V are (chains, L, d); Omega is (M, d).
"""
import numpy as np

from .features import feature_map


def att_lin_quadratic(Q, K, V, Omega, feature):
    """Eq. 2, first form.  Rows whose denominator is exactly 0 (possible only
    for the ReLU map) get output 0."""
    Qt = feature_map(Q, Omega, feature)
    Kt = feature_map(K, Omega, feature)
    chains, L, d = V.shape
    Y = np.zeros((chains, L, d))
    for c in range(chains):
        for l in range(L):
            w = Kt[c, : l + 1] @ Qt[c, l]          # g(K_l')^T g(Q_l), l' = 1..l
            den = w.sum()
            if den != 0.0:
                Y[c, l] = (w[:, None] * V[c, : l + 1]).sum(axis=0) / den
    return Y

