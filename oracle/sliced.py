"""Low-memory forward/backward of one causal linear-attention layer (s = 1), fp64.

ORACLE -- test infrastructure only; see oracle/__init__.py.

This follows Algorithm 1 with its per-slice step (Algorithm 2) for a single
layer whose F computes T_l = [g(K_l), V_l g(K_l)^T] and Gamma_l = g(Q_l)
(Sec. 3.1) and whose G is the division of eq. 4.  The carried state is
B = U_{B_n} = (R, S): R = sum V_l g(K_l)^T (d x M) and S = sum g(K_l) (M),
the last rows of the prefix sums of eq. 3 (Sec. 3.2).

Forward sweep (Sec. 3.2, eqs. 14-16), n = 1..N:
    U := 1 B^T + PS(T);  Y := U_R g(Q) / U_S^T g(Q);  B := U_{B_n}.
Backward sweep (Sec. 3.3), n = N..1, with G^(N) = 0:
    B -= sum_l T_l                                  (eq. 17, rollback)
    U := 1 B^T + PS(T);  Phi := <dY, Y> + <G, U_{B_n}>
    G := grad_B Phi                                 (eq. 18)
and the slice's parameter/input gradients are grad Phi.  The loss of eq. 10
is replaced by <dY, Y> for an upstream cotangent dY, so the gradients are the
vector-Jacobian product of the layer.  Gradients of Phi are written out by the
chain rule (the paper uses autodiff): the gradient of a prefix sum is the
reversed (suffix, inclusive) prefix sum of the output gradient (Sec. 3.3 --
where the paper's index reads "l' = t", it is l' = l).

Inside a slice the whole prefix sum is taken at once (Algorithm 2).  When a
slice is large, it is evaluated in blocks of `block` rows with the running
front carried between blocks, the "block" iteration of App. B; block and
slice recurrences are the same recurrence, so the result is unchanged in
exact arithmetic.

Shapes: Q, K, V, dY are (chains, L, d); Omega is (M, d); R is (chains, d, M);
S is (chains, M).  A denominator that is exactly 0 (ReLU map only) gives a
zero output row and zero gradients for that row.
"""
import math

import numpy as np

from .features import feature_map, feature_vjp

# Slices with more than this many prefix-sum entries (rows * d * M per chain)
# are evaluated block by block (App. B).
_WHOLE_SLICE_LIMIT = 1 << 21
BLOCK = 64  # App. B block size


def _T(Kt, V):
    """T_l = [g(K_l), V_l g(K_l)^T] as the pair (T_S, T_R): (c,b,M), (c,b,d,M)."""
    return Kt, V[:, :, :, None] * Kt[:, :, None, :]


def _readout(U_R, U_S, Qt):
    """Eq. 4: Y_l = (R_l g(Q_l)) / (S_l^T g(Q_l)); returns Y and the denominator."""
    num = np.einsum("cldm,clm->cld", U_R, Qt)
    den = np.einsum("clm,clm->cl", U_S, Qt)
    safe = np.where(den != 0.0, den, 1.0)
    Y = np.where((den != 0.0)[..., None], num / safe[..., None], 0.0)
    return Y, den


def _forward_rows(R, S, Qt, Kt, V):
    """One application of eqs. 14-16 on a run of rows: U = 1 B^T + PS(T)."""
    T_S, T_R = _T(Kt, V)
    U_S = S[:, None, :] + np.cumsum(T_S, axis=1)
    U_R = R[:, None, :, :] + np.cumsum(T_R, axis=1)
    Y, _ = _readout(U_R, U_S, Qt)
    return Y, U_R[:, -1], U_S[:, -1]


def _backward_rows(R, S, G_R, G_S, Qt, Kt, V, dY):
    """Backward step on a run of rows whose end state is B = (R, S) and whose
    incoming state gradient is G = (G_R, G_S).  Returns the feature-space
    gradients, the rolled-back state B^(n-1) and the new G^(n-1)."""
    T_S, T_R = _T(Kt, V)
    # eq. 17: B^(n-1) = B^(n) - sum_l T_l
    R0 = R - T_R.sum(axis=1)
    S0 = S - T_S.sum(axis=1)
    U_S = S0[:, None, :] + np.cumsum(T_S, axis=1)
    U_R = R0[:, None, :, :] + np.cumsum(T_R, axis=1)
    Y, den = _readout(U_R, U_S, Qt)
    # Phi = <dY, Y> + <G_R, U_R[last]> + <G_S, U_S[last]>
    ok = den != 0.0
    safe = np.where(ok, den, 1.0)
    dnum = np.where(ok[..., None], dY / safe[..., None], 0.0)
    dden = np.where(ok, -np.sum(dY * Y, axis=-1) / safe, 0.0)
    dU_R = dnum[:, :, :, None] * Qt[:, :, None, :]
    dU_S = dden[:, :, None] * Qt
    dU_R[:, -1] += G_R
    dU_S[:, -1] += G_S
    dQt = np.einsum("cldm,cld->clm", U_R, dnum) + U_S * dden[:, :, None]
    # gradient through PS: reversed prefix sum (inclusive suffix sum)
    dT_R = np.flip(np.cumsum(np.flip(dU_R, axis=1), axis=1), axis=1)
    dT_S = np.flip(np.cumsum(np.flip(dU_S, axis=1), axis=1), axis=1)
    # eq. 18: G^(n-1) = grad of Phi w.r.t. B^(n-1) = sum_l dU_l = dT_1
    G_R_new = dT_R[:, 0].copy()
    G_S_new = dT_S[:, 0].copy()
    # T_l = [g(K_l), V_l g(K_l)^T]
    dKt = dT_S + np.einsum("cldm,cld->clm", dT_R, V)
    dV = np.einsum("cldm,clm->cld", dT_R, Kt)
    return dQt, dKt, dV, R0, S0, G_R_new, G_S_new


def _row_blocks(b, d, M, block):
    """Split b rows of one slice into runs: the whole slice (Algorithm 2) when it
    is small, else App. B blocks."""
    if block is None:
        block = b if b * d * M <= _WHOLE_SLICE_LIMIT else BLOCK
    return [(s, min(s + block, b)) for s in range(0, b, block)]


def slices(L, C):
    """Slice bounds (A_n, A_n + B_n) for n = 1..N, N = ceil(L/C), A_n = (n-1)C,
    the last slice possibly shorter (Sec. 3.2).  C > L behaves as C = L."""
    if C < 1:
        raise ValueError("C must be >= 1")
    C = min(C, L)
    N = math.ceil(L / C) if L > 0 else 0
    return [((n - 1) * C, min(n * C, L)) for n in range(1, N + 1)]


def forward_features(Qt, Kt, V, C, R0=None, S0=None, block=None):
    """Forward sweep of Algorithm 1 in feature space (g(Q), g(K) given).
    Returns Y, and the final state B^(N) = (R, S)."""
    c, L, d = V.shape
    M = Qt.shape[-1]
    R = np.zeros((c, d, M)) if R0 is None else np.array(R0, dtype=np.float64)
    S = np.zeros((c, M)) if S0 is None else np.array(S0, dtype=np.float64)
    Y = np.zeros((c, L, d))
    for a, e in slices(L, C):
        for s0, s1 in _row_blocks(e - a, d, M, block):
            r = slice(a + s0, a + s1)
            Y[:, r], R, S = _forward_rows(R, S, Qt[:, r], Kt[:, r], V[:, r])
    return Y, R, S


def backward_features(Qt, Kt, V, dY, C, R_N, S_N, G_R=None, G_S=None, block=None):
    """Backward sweep of Algorithm 1 in feature space.  Starts from the final
    state B^(N) = (R_N, S_N) and G^(N) (zero unless given).  Returns
    dL/dg(Q), dL/dg(K), dL/dV, the rolled-back B^(0) and G^(0)."""
    c, L, d = V.shape
    M = Qt.shape[-1]
    R = np.array(R_N, dtype=np.float64)
    S = np.array(S_N, dtype=np.float64)
    G_R = np.zeros((c, d, M)) if G_R is None else np.array(G_R, dtype=np.float64)
    G_S = np.zeros((c, M)) if G_S is None else np.array(G_S, dtype=np.float64)
    dQt = np.zeros_like(Qt)
    dKt = np.zeros_like(Kt)
    dV = np.zeros_like(V)
    for a, e in reversed(slices(L, C)):
        for s0, s1 in reversed(_row_blocks(e - a, d, M, block)):
            r = slice(a + s0, a + s1)
            dQt[:, r], dKt[:, r], dV[:, r], R, S, G_R, G_S = _backward_rows(
                R, S, G_R, G_S, Qt[:, r], Kt[:, r], V[:, r], dY[:, r])
    return dQt, dKt, dV, R, S, G_R, G_S


def forward(Q, K, V, Omega, C, feature, R0=None, S0=None, block=None):
    """Algorithm 1, forward sweep: features are recomputed slice by slice
    (F is applied row-wise).  Returns Y, R^(N), S^(N)."""
    c, L, d = V.shape
    M = Omega.shape[0]
    R = np.zeros((c, d, M)) if R0 is None else np.array(R0, dtype=np.float64)
    S = np.zeros((c, M)) if S0 is None else np.array(S0, dtype=np.float64)
    Y = np.zeros((c, L, d))
    for a, e in slices(L, C):
        r = slice(a, e)
        Qt = feature_map(Q[:, r], Omega, feature)
        Kt = feature_map(K[:, r], Omega, feature)
        Y[:, r], R, S = forward_features(Qt, Kt, V[:, r], e - a, R, S, block)
    return Y, R, S


def backward(Q, K, V, Omega, dY, C, feature, R_N, S_N, G_R=None, G_S=None, block=None):
    """Algorithm 1, backward sweep, n = N..1: recompute the slice's features,
    roll the state back (eq. 17), differentiate Phi, carry G (eq. 18).
    Returns dQ, dK, dV, dOmega, B^(0) = (R, S) and G^(0) = (G_R, G_S)."""
    c, L, d = V.shape
    M = Omega.shape[0]
    R = np.array(R_N, dtype=np.float64)
    S = np.array(S_N, dtype=np.float64)
    G_R = np.zeros((c, d, M)) if G_R is None else np.array(G_R, dtype=np.float64)
    G_S = np.zeros((c, M)) if G_S is None else np.array(G_S, dtype=np.float64)
    dQ = np.zeros_like(Q)
    dK = np.zeros_like(K)
    dV = np.zeros_like(V)
    dOmega = np.zeros_like(Omega)
    for a, e in reversed(slices(L, C)):
        r = slice(a, e)
        Qt = feature_map(Q[:, r], Omega, feature)
        Kt = feature_map(K[:, r], Omega, feature)
        dQt, dKt, dV[:, r], R, S, G_R, G_S = backward_features(
            Qt, Kt, V[:, r], dY[:, r], e - a, R, S, G_R, G_S, block)
        dQ[:, r], dOq = feature_vjp(Q[:, r], Omega, dQt, feature)
        dK[:, r], dOk = feature_vjp(K[:, r], Omega, dKt, feature)
        dOmega += dOq + dOk
    return dQ, dK, dV, dOmega, (R, S), (G_R, G_S)
