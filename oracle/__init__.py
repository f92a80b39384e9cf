"""fp64 CPU oracle for sliced causal linear attention (SLiM, arXiv 2012.11346).

THIS PACKAGE IS TEST INFRASTRUCTURE.  Only tests/, __graft_entry__.smoke() and
bench.py's CPU-baseline / reference leg may import it.  The CUDA library never
calls it and shares no code with it; there is no CPU fallback through here.

Modules
  features   -- the feature maps g (FAVOR+ exp, generalized ReLU) and VJPs
  brute      -- eq. 2 written out row by row (O(L^2))
  sliced     -- Algorithm 1 / Algorithm 2 for one layer: forward sweep, and
                backward sweep with rollback (eq. 17) and G carry (eq. 18)
  iterative  -- the token-by-token recurrence of App. B (C = 1)
  fd         -- central finite differences of <dY, Y>
  bidir      -- the non-causal form (no mask, one global state), two sweeps
  stack      -- s residual layers, Algorithm 1 with one state per layer

Library-facing wrappers below use the layout of the C ABI: q, k, v, dout are
[B, H, L, d]; omega is [M, d]; the state is S_state = R^T ([B, H, M, d], the
sum of g(k) v^T) and z_state = S ([B, H, M], the sum of g(k)) in the paper's
notation of eq. 3.

Parity pins (tests/test_oracle_pins.py): quadratic definition, C-invariance,
App. B recurrence, closed forms (Omega = 0, final state), finite differences,
FAVOR+ / arc-cosine kernel expectations, rollback closure B^(0) = 0.  No
function here is "parity unpinned".
"""
import numpy as np

from . import bidir, brute, features, fd, iterative, sliced, stack  # noqa: F401


def _chains(x):
    x = np.asarray(x, dtype=np.float64)
    B, H, L, d = x.shape
    return x.reshape(B * H, L, d), (B, H)


def oracle_fwd(q, k, v, omega, C, feature, S0=None, z0=None):
    """Forward sweep.  Returns out [B,H,L,d], S_state [B,H,M,d], z_state [B,H,M]."""
    Q, (B, H) = _chains(q)
    K, _ = _chains(k)
    V, _ = _chains(v)
    Omega = np.asarray(omega, dtype=np.float64)
    M = Omega.shape[0]
    R0 = None if S0 is None else np.swapaxes(np.asarray(S0, np.float64).reshape(B * H, M, -1), 1, 2)
    Si = None if z0 is None else np.asarray(z0, np.float64).reshape(B * H, M)
    Y, R, S = sliced.forward(Q, K, V, Omega, C, feature, R0, Si)
    L, d = Q.shape[1], Q.shape[2]
    return (Y.reshape(B, H, L, d),
            np.swapaxes(R, 1, 2).reshape(B, H, M, d),
            S.reshape(B, H, M))


def oracle_bwd(q, k, v, omega, dout, S_state, z_state, C, feature, G_S=None, g_z=None):
    """Backward sweep from B^(N) = (S_state, z_state), with the state gradient
    G^(N) = (G_S, g_z) handed in by a later segment (zero if None; Sec. 3.3).
    Returns dq, dk, dv ([B,H,L,d]), domega ([M,d]) and a dict with the
    rolled-back state B^(0) and the state gradient G^(0) (same layout as
    S_state / z_state)."""
    Q, (B, H) = _chains(q)
    K, _ = _chains(k)
    V, _ = _chains(v)
    dY, _ = _chains(dout)
    Omega = np.asarray(omega, dtype=np.float64)
    M = Omega.shape[0]
    L, d = Q.shape[1], Q.shape[2]
    R_N = np.swapaxes(np.asarray(S_state, np.float64).reshape(B * H, M, d), 1, 2)
    S_N = np.asarray(z_state, np.float64).reshape(B * H, M)
    G_R_N = None if G_S is None else np.swapaxes(np.asarray(G_S, np.float64).reshape(B * H, M, d), 1, 2)
    G_S_N = None if g_z is None else np.asarray(g_z, np.float64).reshape(B * H, M)
    dQ, dK, dV, dOmega, (R0, S0), (G_R, G_S) = sliced.backward(
        Q, K, V, Omega, dY, C, feature, R_N, S_N, G_R_N, G_S_N)
    extra = {
        "S0": np.swapaxes(R0, 1, 2).reshape(B, H, M, d),
        "z0": S0.reshape(B, H, M),
        "G_S": np.swapaxes(G_R, 1, 2).reshape(B, H, M, d),
        "g_z": G_S.reshape(B, H, M),
    }
    return (dQ.reshape(B, H, L, d), dK.reshape(B, H, L, d), dV.reshape(B, H, L, d),
            dOmega, extra)


def oracle_bidir_fwd(q, k, v, omega, C, feature):
    """Non-causal forward.  Returns out [B,H,L,d], S_state [B,H,M,d], z_state
    [B,H,M] (the global state)."""
    Q, (B, H) = _chains(q)
    K, _ = _chains(k)
    V, _ = _chains(v)
    Omega = np.asarray(omega, dtype=np.float64)
    M = Omega.shape[0]
    L, d = Q.shape[1], Q.shape[2]
    Y, R, S = bidir.forward(Q, K, V, Omega, C, feature)
    return (Y.reshape(B, H, L, d), np.swapaxes(R, 1, 2).reshape(B, H, M, d), S.reshape(B, H, M))


def oracle_bidir_bwd(q, k, v, omega, dout, S_state, z_state, C, feature):
    """Non-causal backward from the global state.  Returns dq, dk, dv, domega."""
    Q, (B, H) = _chains(q)
    K, _ = _chains(k)
    V, _ = _chains(v)
    dY, _ = _chains(dout)
    Omega = np.asarray(omega, dtype=np.float64)
    M = Omega.shape[0]
    L, d = Q.shape[1], Q.shape[2]
    R = np.swapaxes(np.asarray(S_state, np.float64).reshape(B * H, M, d), 1, 2)
    S = np.asarray(z_state, np.float64).reshape(B * H, M)
    dQ, dK, dV, dOmega, _ = bidir.backward(Q, K, V, Omega, dY, C, feature, R, S)
    return (dQ.reshape(B, H, L, d), dK.reshape(B, H, L, d), dV.reshape(B, H, L, d), dOmega)


def oracle_stack_fwd(x, omegas, C, feature):
    """Stack forward: x [B,H,L,d], omegas [s][M,d].  Returns y [B,H,L,d] and the
    final states S_state [s][B,H,M,d], z_state [s][B,H,M]."""
    X, (B, H) = _chains(x)
    Oms = [np.asarray(o, dtype=np.float64) for o in omegas]
    L, d = X.shape[1], X.shape[2]
    Y, states = stack.forward(X, Oms, C, feature)
    S = np.stack([np.swapaxes(R, 1, 2).reshape(B, H, Om.shape[0], d) for (R, _), Om in zip(states, Oms)])
    z = np.stack([Sz.reshape(B, H, Om.shape[0]) for (_, Sz), Om in zip(states, Oms)])
    return Y.reshape(B, H, L, d), S, z


def oracle_stack_bwd(x, omegas, dy, S_state, z_state, C, feature):
    """Stack backward from the final states.  Returns dx [B,H,L,d] and
    domegas [s][M,d]."""
    X, (B, H) = _chains(x)
    dY, _ = _chains(dy)
    Oms = [np.asarray(o, dtype=np.float64) for o in omegas]
    L, d = X.shape[1], X.shape[2]
    states = [(np.swapaxes(np.asarray(S_state[r], np.float64).reshape(B * H, Om.shape[0], d), 1, 2),
               np.asarray(z_state[r], np.float64).reshape(B * H, Om.shape[0]))
              for r, Om in enumerate(Oms)]
    dX, dOm, _ = stack.backward(X, Oms, dY, C, feature, states)
    return dX.reshape(B, H, L, d), np.stack(dOm)


def rel_l2(a, b):
    """||a - b||_2 / ||b||_2 over the whole tensor (the discrepancy measure of
    Sec. 4.2)."""
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    if not (np.all(np.isfinite(a)) and np.all(np.isfinite(b))):
        return float("inf")
    nb = np.linalg.norm(b.ravel())
    return float(np.linalg.norm((a - b).ravel()) / (nb if nb > 0 else 1.0))
