"""A stack of s causal linear-attention layers evaluated the memory-efficient
way of Algorithm 1, fp64.

ORACLE -- test infrastructure only; see oracle/__init__.py.

Layer r (r = 1..s) maps each row of its input X^(r-1) to a query, a key and a
value -- all three the row normalised to a fixed root-mean-square,

    u = d^(-1/4) x / sqrt(mean_i x_i^2 + eps),       q = k = v = u,

a parameter-free stand-in for the row-wise layer normalisation of the paper's
model (Sec. 2.2, eqs. 5-6) that keeps every layer's features at the scale of the
single-layer inputs -- runs the causal linear attention of eq. 2 on them with
its own random-feature matrix Omega_r, and adds the result back (a residual
connection):

    X^(r) = X^(r-1) + Att_r(u(X^(r-1)), u(X^(r-1)), u(X^(r-1))),   r = 1..s.

That is the F / prefix sum / G split of Sec. 3.1 (eqs. 11-13) with F^(r)
computing T = (V g(K)^T, g(K)) and Gamma = g(Q) from the row, and G^(r) the
readout of eq. 4 plus the residual add.  The output is X^(s); the objective
whose gradient is taken is <dY, X^(s)> for an upstream cotangent dY.

Algorithm 1 keeps one state per layer, B_r = (R_r, S_r) (the matrix of s rows
of Sec. 3.2), walks the slices in the outer loop and the layers in the inner
loop (Algorithm 2):
  forward, n = 1..N:  X := X^(0) rows of slice n;  for r = 1..s:
      Y, B_r := layer r on the slice from B_r;  X := X + Y
  backward, n = N..1, G_r = 0 at the start (eq. 18):
      recompute the slice layer by layer: for r = 1..s: B_r -= sum of the
      slice's T_l (eq. 17, the keys of layer r on this slice need the
      rolled-back states of layers < r first), keep X^(r-1) of the slice
      and recompute layer r's output;
      then for r = s..1: the slice's gradients of layer r from its saved input,
      its final state B_r^(n) and G_r; G_r := the gradient with respect to
      B_r^(n-1); dX^(r-1) = dX^(r) + u'(X^(r-1))^T (dq + dk + dv) (the residual,
      and q = k = v = u(X^(r-1))).
Only the s states, their gradients and one slice's activations are kept:
O(C) memory besides the input (Sec. 3.4).

Shapes: X, dY are (chains, L, d); Omegas is a list of s (M, d) arrays.
"""
import numpy as np

from . import brute
from .sliced import backward as layer_backward
from .sliced import forward as layer_forward
from .sliced import slices

EPS = 1e-6


def row_norm(X):
    """u = d^(-1/4) x / sqrt(mean(x^2) + eps), row by row."""
    d = X.shape[-1]
    r = np.sqrt(np.mean(X * X, axis=-1, keepdims=True) + EPS)
    return d ** -0.25 * X / r


def row_norm_vjp(X, g):
    """Cotangent g of u = row_norm(x) pulled back to x:
    dx = (s / r) (g - x mean(g x) / r^2), s = d^(-1/4)."""
    d = X.shape[-1]
    r = np.sqrt(np.mean(X * X, axis=-1, keepdims=True) + EPS)
    return d ** -0.25 / r * (g - X * np.mean(g * X, axis=-1, keepdims=True) / (r * r))


def quadratic(X0, Omegas, feature):
    """The stack layer by layer over the whole sequence, each layer by the
    row-by-row definition of eq. 2 (tiny inputs)."""
    X = np.array(X0, dtype=np.float64)
    for Om in Omegas:
        U = row_norm(X)
        X = X + brute.att_lin_quadratic(U, U, U, Om, feature)
    return X


def forward(X0, Omegas, C, feature):
    """Algorithm 1's forward sweep for the stack.  Returns X^(s) and the final
    states [(R_r, S_r)] of every layer."""
    c, L, d = X0.shape
    states = [(np.zeros((c, d, Om.shape[0])), np.zeros((c, Om.shape[0]))) for Om in Omegas]
    Y = np.zeros((c, L, d))
    for a, e in slices(L, C):
        X = np.array(X0[:, a:e], dtype=np.float64)
        for r, Om in enumerate(Omegas):
            R, S = states[r]
            U = row_norm(X)
            out, R, S = layer_forward(U, U, U, Om, e - a, feature, R, S)
            states[r] = (R, S)
            X = X + out
        Y[:, a:e] = X
    return Y, states


def backward(X0, Omegas, dY, C, feature, states):
    """Algorithm 1's backward sweep for the stack, from the final states the
    forward returned.  Returns dX^(0), [dOmega_r] and the rolled-back states
    (zero when the rollback closes)."""
    c, L, d = X0.shape
    s = len(Omegas)
    B = [(np.array(R), np.array(S)) for R, S in states]
    G = [(np.zeros_like(R), np.zeros_like(S)) for R, S in B]
    dX0 = np.zeros((c, L, d))
    dOm = [np.zeros_like(Om, dtype=np.float64) for Om in Omegas]
    for a, e in reversed(slices(L, C)):
        # recompute the slice, layer by layer, rolling each state back (eq. 17)
        ins, ends = [], []
        X = np.array(X0[:, a:e], dtype=np.float64)
        for r, Om in enumerate(Omegas):
            R_end, S_end = B[r]
            U = row_norm(X)
            # the slice's own contribution, sum of T_l over its rows
            _, dR, dS = layer_forward(U, U, U, Om, e - a, feature)
            B[r] = (R_end - dR, S_end - dS)
            out, _, _ = layer_forward(U, U, U, Om, e - a, feature, B[r][0], B[r][1])
            ins.append(X)
            ends.append((R_end, S_end))
            X = X + out
        # back through the layers: the residual passes dX on; q = k = v = u(X)
        dX = np.array(dY[:, a:e], dtype=np.float64)
        for r in reversed(range(s)):
            Xr = ins[r]
            U = row_norm(Xr)
            dq, dk, dv, dO, _, G[r] = layer_backward(U, U, U, Omegas[r], dX, e - a, feature,
                                                     ends[r][0], ends[r][1], G[r][0], G[r][1])
            dOm[r] += dO
            dX = dX + row_norm_vjp(Xr, dq + dk + dv)
        dX0[:, a:e] = dX
    return dX0, dOm, B
