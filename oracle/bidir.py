"""Non-causal (bidirectional) linear attention, fp64.

ORACLE -- test infrastructure only; see oracle/__init__.py.

Eq. 2 without the causal mask: every position reads every key,

    Y_l = sum_{l'=1..L} V_l' (g(K_l')^T g(Q_l)) / sum_{l'=1..L} g(K_l')^T g(Q_l),

so one global state B = (R, S) = (sum_l V_l g(K_l)^T, sum_l g(K_l)) serves every row
(eq. 3 at l = L).  The paper treats the causal form only (Sec. 2.1); this is the
same computation with the prefix sums replaced by the full sum.  Memory stays
O(C) the same way Algorithm 1 keeps it: the sequence is read slice by slice,
twice -- the first sweep accumulates B, the second reads it out -- and the
backward sweeps the slices twice as well: first the query side, which also
accumulates the state gradient G = grad_B <dY, Y>, then the key/value side,
which reads G.

Shapes as in sliced.py: Q, K, V, dY are (chains, L, d); Omega is (M, d);
R is (chains, d, M); S is (chains, M).
"""
import numpy as np

from .features import feature_map, feature_vjp
from .sliced import slices


def quadratic(Q, K, V, Omega, feature):
    """The definition above, row by row (O(L^2)), for tiny inputs.  A row whose
    denominator is exactly 0 gets output 0."""
    Qt = feature_map(Q, Omega, feature)
    Kt = feature_map(K, Omega, feature)
    chains, L, d = V.shape
    Y = np.zeros((chains, L, d))
    for c in range(chains):
        for l in range(L):
            w = Kt[c] @ Qt[c, l]
            den = w.sum()
            if den != 0.0:
                Y[c, l] = (w[:, None] * V[c]).sum(axis=0) / den
    return Y


def _readout(R, S, Qt):
    num = np.einsum("cdm,clm->cld", R, Qt)
    den = np.einsum("cm,clm->cl", S, Qt)
    ok = den != 0.0
    safe = np.where(ok, den, 1.0)
    return np.where(ok[..., None], num / safe[..., None], 0.0), den


def forward(Q, K, V, Omega, C, feature):
    """Two sweeps over slices of C rows: B = sum of T_l, then Y = readout.
    Returns Y, R, S."""
    c, L, d = V.shape
    M = Omega.shape[0]
    R = np.zeros((c, d, M))
    S = np.zeros((c, M))
    for a, e in slices(L, C):
        Kt = feature_map(K[:, a:e], Omega, feature)
        R += np.einsum("cld,clm->cdm", V[:, a:e], Kt)
        S += Kt.sum(axis=1)
    Y = np.zeros((c, L, d))
    for a, e in slices(L, C):
        Qt = feature_map(Q[:, a:e], Omega, feature)
        Y[:, a:e], _ = _readout(R, S, Qt)
    return Y, R, S


def backward(Q, K, V, Omega, dY, C, feature, R, S):
    """Gradients of <dY, Y> from the global state (R, S) the forward returned.
    Sweep 1 (query side), per slice: den, dnum = dY/den, dden = -<dY, Y>/den,
    dg(Q) = R^T dnum + S dden, and G_R += dnum g(Q)^T, G_S += dden g(Q).
    Sweep 2 (key/value side), per slice: dg(K) = G_R^T V + G_S, dV = G_R g(K).
    Returns dQ, dK, dV, dOmega and G = (G_R, G_S)."""
    c, L, d = V.shape
    M = Omega.shape[0]
    G_R = np.zeros((c, d, M))
    G_S = np.zeros((c, M))
    dQ = np.zeros_like(Q)
    dK = np.zeros_like(K)
    dV = np.zeros_like(V)
    dOmega = np.zeros_like(Omega, dtype=np.float64)
    for a, e in slices(L, C):
        Qt = feature_map(Q[:, a:e], Omega, feature)
        Y, den = _readout(R, S, Qt)
        ok = den != 0.0
        safe = np.where(ok, den, 1.0)
        dnum = np.where(ok[..., None], dY[:, a:e] / safe[..., None], 0.0)
        dden = np.where(ok, -np.sum(dY[:, a:e] * Y, axis=-1) / safe, 0.0)
        dQt = np.einsum("cdm,cld->clm", R, dnum) + S[:, None, :] * dden[..., None]
        G_R += np.einsum("cld,clm->cdm", dnum, Qt)
        G_S += np.einsum("cl,clm->cm", dden, Qt)
        dQ[:, a:e], dOq = feature_vjp(Q[:, a:e], Omega, dQt, feature)
        dOmega += dOq
    for a, e in slices(L, C):
        Kt = feature_map(K[:, a:e], Omega, feature)
        dKt = np.einsum("cdm,cld->clm", G_R, V[:, a:e]) + G_S[:, None, :]
        dV[:, a:e] = np.einsum("cdm,clm->cld", G_R, Kt)
        dK[:, a:e], dOk = feature_vjp(K[:, a:e], Omega, dKt, feature)
        dOmega += dOk
    return dQ, dK, dV, dOmega, (G_R, G_S)
