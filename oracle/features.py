"""Feature maps g: R^d -> R_+^M of causal linear attention, and their VJPs (fp64).

ORACLE -- test infrastructure only.  Nothing in the product path may import this
module; only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg do.

The paper (Sec. 2.1, eq. 2) leaves g abstract: a map into vectors with positive
entries, M features per d-dimensional input.  Two instances are used here:

* FAVOR+ positive random features (the randomized g the paper cites in Sec. 2.1):
      g(x)_m = exp(omega_m . x - |x|^2 / 2) / sqrt(M)
  No max-stabiliser and no epsilon (the inputs keep omega.x well inside fp32
  range).
* generalized ReLU random features:
      g(x)_m = max(omega_m . x, 0) / sqrt(M)
  with ReLU'(0) = 0.
* the elementwise quadratic map of the paper's experiments (Sec. 4, with
  M = d, and Sec. 2.1's remark that g can be elementwise):
      g(x)_i = x_i^2,   i = 1..d
  It has no random features: Omega is not used (only its shape, M = d, is
  checked) and its gradient is zero.

Omega is M x d and shared by every (batch, head) chain; its gradient is the sum
over all chains and over both the query and the key side.

Arrays are float64.  X has shape (..., L, d), g(X) has shape (..., L, M).
"""
import numpy as np

FEATURES = ("exp", "relu", "square")


def projection(X, Omega):
    """omega_m . x for every row x of X: (..., L, d) x (M, d) -> (..., L, M)."""
    return np.einsum("...ld,md->...lm", X, Omega)


def g_exp(X, Omega):
    """FAVOR+ map exp(Omega x - |x|^2/2)/sqrt(M), row by row."""
    M = Omega.shape[0]
    half_sq = 0.5 * np.sum(X * X, axis=-1, keepdims=True)
    return np.exp(projection(X, Omega) - half_sq) / np.sqrt(M)


def g_relu(X, Omega):
    """Generalized-ReLU map max(Omega x, 0)/sqrt(M), row by row."""
    M = Omega.shape[0]
    return np.maximum(projection(X, Omega), 0.0) / np.sqrt(M)


def g_square(X, Omega):
    """Elementwise quadratic map (x_1^2, ..., x_d^2); M = d."""
    if Omega.shape[0] != X.shape[-1]:
        raise ValueError("the quadratic map has M = d features")
    return X * X


def feature_map(X, Omega, feature):
    if feature == "exp":
        return g_exp(X, Omega)
    if feature == "relu":
        return g_relu(X, Omega)
    if feature == "square":
        return g_square(X, Omega)
    raise ValueError(f"unknown feature map {feature!r}")


def feature_vjp(X, Omega, dG, feature):
    """Pull the cotangent dG = dL/dg(X) back to (dL/dX, dL/dOmega).

    exp:  dg_m/dx = g_m (omega_m - x)        -> u = dG*g,
          dX = u Omega - x sum_m u_m,  dOmega = sum_rows u^T x
    relu: dg_m/dx = 1[omega_m.x > 0] omega_m / sqrt(M)
                                              -> u = dG*1[.>0]/sqrt(M),
          dX = u Omega,                dOmega = sum_rows u^T x
    square: dg_i/dx_i = 2 x_i (and 0 off the diagonal)
                                              -> dX = 2 x * dG,  dOmega = 0
    dOmega is summed over every leading axis (all chains, all rows).
    """
    if feature == "square":
        g_square(X, Omega)  # shape check
        return 2.0 * X * dG, np.zeros_like(Omega, dtype=np.float64)
    M = Omega.shape[0]
    if feature == "exp":
        u = dG * g_exp(X, Omega)
        dX = np.einsum("...lm,md->...ld", u, Omega) - X * np.sum(u, axis=-1, keepdims=True)
    elif feature == "relu":
        u = dG * (projection(X, Omega) > 0.0) / np.sqrt(M)
        dX = np.einsum("...lm,md->...ld", u, Omega)
    else:
        raise ValueError(f"unknown feature map {feature!r}")
    dOmega = u.reshape(-1, M).T @ X.reshape(-1, X.shape[-1])
    return dX, dOmega
