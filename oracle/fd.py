"""Central finite differences of the scalar <dY, Y(Q, K, V, Omega)>, fp64.

ORACLE -- test infrastructure only; see oracle/__init__.py.

Y is the quadratic definition of eq. 2 (brute.att_lin_quadratic), so these
derivatives are independent of the sliced backward sweep they check.
"""
import numpy as np

from .brute import att_lin_quadratic


def _objective(Q, K, V, Omega, dY, feature, fn=att_lin_quadratic):
    return float(np.sum(dY * fn(Q, K, V, Omega, feature)))


def central_differences(Q, K, V, Omega, dY, feature, h=1e-6, fn=att_lin_quadratic):
    """Returns (dQ, dK, dV, dOmega) by (f(x+h e_i) - f(x-h e_i)) / 2h, f the
    scalar <dY, fn(Q, K, V, Omega)> (eq. 2 by default)."""
    args = [np.array(a, dtype=np.float64) for a in (Q, K, V, Omega)]
    grads = []
    for which in range(4):
        x = args[which]
        g = np.zeros_like(x)
        it = np.nditer(x, flags=["multi_index"])
        for _ in it:
            idx = it.multi_index
            keep = x[idx]
            x[idx] = keep + h
            fp = _objective(*args, dY, feature, fn)
            x[idx] = keep - h
            fm = _objective(*args, dY, feature, fn)
            x[idx] = keep
            g[idx] = (fp - fm) / (2.0 * h)
        grads.append(g)
    return tuple(grads)


def central_differences_initial_state(Qt, Kt, V, dY, R0, S0, forward_features, h=1e-6):
    """d<dY, Y>/dB^(0) for the feature-space forward sweep started from an
    initial state B^(0) = (R0, S0); used to pin G^(0) of the backward sweep."""
    def f(R, S):
        Y, _, _ = forward_features(Qt, Kt, V, V.shape[1], R, S)
        return float(np.sum(dY * Y))

    gR = np.zeros_like(R0)
    gS = np.zeros_like(S0)
    for arr, g in ((R0, gR), (S0, gS)):
        it = np.nditer(arr, flags=["multi_index"])
        for _ in it:
            idx = it.multi_index
            keep = arr[idx]
            arr[idx] = keep + h
            fp = f(R0, S0)
            arr[idx] = keep - h
            fm = f(R0, S0)
            arr[idx] = keep
            g[idx] = (fp - fm) / (2.0 * h)
    return gR, gS
