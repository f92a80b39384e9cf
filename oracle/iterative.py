"""Token-by-token recurrence of App. B (the C = 1 limit of Algorithm 1), fp64.

ORACLE -- test infrastructure only; see oracle/__init__.py.

Forward: buffers curR (d x M) and curS (M) start at zero; for each position l
the key's contribution is added first and then the query reads the buffers,
so the mask is inclusive.  N_l = curR g(Q_l), D_l = curS^T g(Q_l),
Y_l = N_l / D_l.

Backward: start from the forward's final buffers, with gradient buffers
gradR = 0, gradS = 0, and walk l = L..1.  The query gradient reads the
buffers before the key's contribution is removed; the value/key gradients read
the gradient buffers after the query's contribution is added.  App. B lists
only the numerator's share of the key gradient; the normaliser D also depends
on g(K_l) through curS, so its share, gradS, is added here.

Everything is in feature space: Qt = g(Q), Kt = g(K), shapes (L, M); V, dY
are (L, d).  One chain at a time; plain Python loops, so tiny inputs only.
"""
import numpy as np


def forward(Qt, Kt, V):
    L, d = V.shape
    M = Qt.shape[1]
    curR = np.zeros((d, M))
    curS = np.zeros(M)
    Y = np.zeros((L, d))
    for l in range(L):
        curR = curR + np.outer(V[l], Kt[l])
        curS = curS + Kt[l]
        N_l = curR @ Qt[l]
        D_l = curS @ Qt[l]
        Y[l] = N_l / D_l
    return Y, curR, curS


def backward(Qt, Kt, V, dY, curR, curS):
    """dY is the cotangent of Y; returns dL/dg(Q), dL/dg(K), dL/dV and the
    buffers after the walk (which should be back at zero)."""
    L, d = V.shape
    M = Qt.shape[1]
    # cotangents of N and D from Y = N / D
    Y = np.zeros((L, d))
    D = np.zeros(L)
    R, S = curR.copy(), curS.copy()
    for l in reversed(range(L)):
        D[l] = S @ Qt[l]
        Y[l] = (R @ Qt[l]) / D[l]
        R = R - np.outer(V[l], Kt[l])
        S = S - Kt[l]
    gN = dY / D[:, None]
    gD = -np.sum(dY * Y, axis=1) / D

    gradR = np.zeros((d, M))
    gradS = np.zeros(M)
    dQt = np.zeros((L, M))
    dKt = np.zeros((L, M))
    dV = np.zeros((L, d))
    for l in reversed(range(L)):
        dQt[l] = gD[l] * curS + curR.T @ gN[l]
        curR = curR - np.outer(V[l], Kt[l])
        curS = curS - Kt[l]
        gradR = gradR + np.outer(gN[l], Qt[l])
        gradS = gradS + gD[l] * Qt[l]
        dV[l] = gradR @ Kt[l]
        dKt[l] = gradR.T @ V[l] + gradS
    return dQt, dKt, dV, curR, curS
