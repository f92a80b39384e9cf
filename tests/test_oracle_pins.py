"""Pins of the fp64 oracle to facts outside itself (CPU only).

Each pin is a function returning an error measure, so tests/test_oracle_mutations.py
can plant a mistake in the oracle and show that some pin catches it.
"""
import json
import math
import os

import numpy as np
import pytest

import oracle
from oracle import brute, fd, features, iterative, sliced

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "hand_examples.json")


def rel(a, b):
    return oracle.rel_l2(a, b)


def small_case(seed, chains=2, L=40, d=4, M=None, feature="exp", scale=None):
    """Random fp64 inputs.  The ReLU map gets more features so that no row has
    an all-zero weight vector (eq. 2 needs a positive denominator)."""
    rng = np.random.default_rng(seed)
    if feature == "square":
        M = d            # the elementwise map has one feature per input coordinate
    elif M is None:
        M = 6 if feature == "exp" else 24
    s = d ** -0.25 if scale is None else scale
    if feature == "relu":
        Q = rng.uniform(-1, 1, (chains, L, d))
        K = rng.uniform(-1, 1, (chains, L, d))
        V = rng.uniform(-1, 1, (chains, L, d))
    else:
        Q = rng.standard_normal((chains, L, d)) * s
        K = rng.standard_normal((chains, L, d)) * s
        V = rng.standard_normal((chains, L, d)) * s
    Omega = rng.standard_normal((M, d))
    dY = rng.standard_normal((chains, L, d))
    return Q, K, V, Omega, dY


# ----------------------------------------------------------------------------- pins

def pin_brute_vs_sliced(feature, Cs=(1, 3, 7, 16, 40, 64)):
    """Eq. 2 (quadratic definition) against Algorithm 1's forward sweep for
    several slice sizes, including 1, a non-divisor of L, L and C > L."""
    Q, K, V, Omega, _ = small_case(1, feature=feature)
    Yb = brute.att_lin_quadratic(Q, K, V, Omega, feature)
    return max(rel(sliced.forward(Q, K, V, Omega, C, feature)[0], Yb) for C in Cs)


def pin_zero_omega_closed_form():
    """Omega = 0 with the exp map: g(x) = exp(-|x|^2/2)/sqrt(M) * 1, so the
    output is the causal average of v_j weighted by w_j = exp(-|k_j|^2/2),
    independent of q."""
    Q, K, V, _, _ = small_case(2, chains=1, L=30)
    Omega = np.zeros((5, Q.shape[-1]))
    Y, _, _ = sliced.forward(Q, K, V, Omega, 7, "exp")
    w = np.exp(-0.5 * np.sum(K[0] ** 2, axis=1))
    expect = np.zeros_like(V[0])
    acc_num = np.zeros(V.shape[-1])
    acc_den = 0.0
    for j in range(V.shape[1]):
        acc_num = acc_num + w[j] * V[0, j]
        acc_den += w[j]
        expect[j] = acc_num / acc_den
    return rel(Y[0], expect)


def pin_final_state_closed_form(feature):
    """B^(N) = last row of the prefix sums (eq. 3): R = V^T g(K), S = sum g(K)."""
    Q, K, V, Omega, _ = small_case(3, feature=feature)
    _, R, S = sliced.forward(Q, K, V, Omega, 9, feature)
    Kt = features.feature_map(K, Omega, feature)
    R_cf = np.einsum("cld,clm->cdm", V, Kt)
    S_cf = Kt.sum(axis=1)
    return max(rel(R, R_cf), rel(S, S_cf))


def pin_recurrence_forward(feature, Cs=(1, 5, 40)):
    """App. B token-by-token recurrence (C = 1 limit) against the sliced sweep."""
    Q, K, V, Omega, _ = small_case(4, chains=1, feature=feature)
    Qt = features.feature_map(Q, Omega, feature)[0]
    Kt = features.feature_map(K, Omega, feature)[0]
    Yi, Ri, Si = iterative.forward(Qt, Kt, V[0])
    err = 0.0
    for C in Cs:
        Y, R, S = sliced.forward(Q, K, V, Omega, C, feature)
        err = max(err, rel(Y[0], Yi), rel(R[0], Ri), rel(S[0], Si))
    return err


def pin_recurrence_backward(feature, Cs=(1, 5, 40)):
    """App. B backward recurrence (with the normaliser's share of the key
    gradient) against the sliced backward sweep, in feature space."""
    Q, K, V, Omega, dY = small_case(5, chains=1, feature=feature)
    Qt = features.feature_map(Q, Omega, feature)
    Kt = features.feature_map(K, Omega, feature)
    _, Ri, Si = iterative.forward(Qt[0], Kt[0], V[0])
    dQi, dKi, dVi, _, _ = iterative.backward(Qt[0], Kt[0], V[0], dY[0], Ri, Si)
    err = 0.0
    for C in Cs:
        _, R, S = sliced.forward_features(Qt, Kt, V, C)
        dQt, dKt, dV, _, _, _, _ = sliced.backward_features(Qt, Kt, V, dY, C, R, S)
        err = max(err, rel(dQt[0], dQi), rel(dKt[0], dKi), rel(dV[0], dVi))
    return err


def pin_finite_differences(feature, C=2):
    """Central differences of <dY, Y> (eq. 2) against the sliced backward sweep."""
    Q, K, V, Omega, dY = small_case(6, chains=1, L=7, d=3, M=5, feature=feature)
    _, R, S = sliced.forward(Q, K, V, Omega, C, feature)
    dQ, dK, dV, dO, _, _ = sliced.backward(Q, K, V, Omega, dY, C, feature, R, S)
    fQ, fK, fV, fO = fd.central_differences(Q, K, V, Omega, dY, feature)
    return max(rel(dQ, fQ), rel(dK, fK), rel(dV, fV), rel(dO, fO))


def pin_rollback_closes(feature):
    """After the reverse walk the rolled-back state is B^(0) = 0 (eq. 17 undoes
    every slice's addition)."""
    Q, K, V, Omega, dY = small_case(7, feature=feature)
    _, R, S = sliced.forward(Q, K, V, Omega, 6, feature)
    *_, (R0, S0), _ = sliced.backward(Q, K, V, Omega, dY, 6, feature, R, S)
    return max(np.abs(R0).max() / np.abs(R).max(), np.abs(S0).max() / np.abs(S).max())


def pin_initial_state_gradient():
    """G^(0) from the backward sweep equals the derivative of <dY, Y> with
    respect to an initial state B^(0) (App. A: G^(n) = grad_{B^(n)} L)."""
    rng = np.random.default_rng(8)
    L, d, M = 6, 2, 3
    Qt = rng.uniform(0.2, 1.0, (1, L, M))
    Kt = rng.uniform(0.2, 1.0, (1, L, M))
    V = rng.standard_normal((1, L, d))
    dY = rng.standard_normal((1, L, d))
    R0 = rng.standard_normal((1, d, M)) * 0.1
    S0 = rng.uniform(0.5, 1.0, (1, M))
    _, RN, SN = sliced.forward_features(Qt, Kt, V, 2, R0, S0)
    *_, G_R, G_S = sliced.backward_features(Qt, Kt, V, dY, 2, RN, SN)
    fR, fS = fd.central_differences_initial_state(Qt, Kt, V, dY, R0.copy(), S0.copy(),
                                                  sliced.forward_features)
    return max(rel(G_R, fR), rel(G_S, fS))


def pin_streaming_continuation(feature):
    """Running the second part of a sequence from the state left by the first
    part reproduces the full run (eqs. 14-16 with B^(n-1) carried)."""
    Q, K, V, Omega, _ = small_case(9, feature=feature)
    a = 17
    Y, R, S = sliced.forward(Q, K, V, Omega, 8, feature)
    _, R1, S1 = sliced.forward(Q[:, :a], K[:, :a], V[:, :a], Omega, 8, feature)
    Y2, R2, S2 = sliced.forward(Q[:, a:], K[:, a:], V[:, a:], Omega, 8, feature, R1, S1)
    return max(rel(Y2, Y[:, a:]), rel(R2, R), rel(S2, S))


def pin_favor_unbiased(M=400000):
    """FAVOR+ property: E_omega[g(q)^T g(k)] = exp(q^T k) for iid N(0, I)
    rows (Monte Carlo, returns the largest relative deviation)."""
    rng = np.random.default_rng(10)
    d = 3
    Omega = rng.standard_normal((M, d))
    worst = 0.0
    for _ in range(3):
        q = rng.standard_normal(d) * 0.4
        k = rng.standard_normal(d) * 0.4
        est = float(features.g_exp(q[None], Omega)[0] @ features.g_exp(k[None], Omega)[0])
        worst = max(worst, abs(est / math.exp(q @ k) - 1.0))
    return worst


def pin_relu_arccos(M=400000):
    """Generalized ReLU map: E[g(q)^T g(k)] = |q||k|(sin t + (pi - t) cos t)/(2 pi),
    t the angle between q and k (arc-cosine kernel of order 1)."""
    rng = np.random.default_rng(11)
    d = 3
    Omega = rng.standard_normal((M, d))
    worst = 0.0
    for _ in range(3):
        q = rng.standard_normal(d)
        k = rng.standard_normal(d)
        nq, nk = np.linalg.norm(q), np.linalg.norm(k)
        t = math.acos(np.clip(q @ k / (nq * nk), -1, 1))
        expect = nq * nk * (math.sin(t) + (math.pi - t) * math.cos(t)) / (2 * math.pi)
        est = float(features.g_relu(q[None], Omega)[0] @ features.g_relu(k[None], Omega)[0])
        worst = max(worst, abs(est / expect - 1.0))
    return worst


def pin_block_equals_whole(feature):
    """App. B block evaluation inside a slice equals the whole-slice prefix sum."""
    Q, K, V, Omega, dY = small_case(12, feature=feature)
    Y1, R1, S1 = sliced.forward(Q, K, V, Omega, 40, feature, block=None)
    Y2, R2, S2 = sliced.forward(Q, K, V, Omega, 40, feature, block=3)
    g1 = sliced.backward(Q, K, V, Omega, dY, 40, feature, R1, S1, block=None)
    g2 = sliced.backward(Q, K, V, Omega, dY, 40, feature, R2, S2, block=3)
    return max([rel(Y2, Y1), rel(R2, R1)] + [rel(a, b) for a, b in zip(g2[:4], g1[:4])])


def pin_golden():
    """Hand-worked examples (eq. 2 and eq. 3)."""
    with open(GOLDEN) as f:
        data = json.load(f)
    worst = 0.0
    for ex in data["examples"]:
        q = np.array(ex["q"])[None, None]
        k = np.array(ex["k"])[None, None]
        v = np.array(ex["v"])[None, None]
        om = np.array(ex["omega"])
        L = q.shape[2]
        for C in (1, 2, L):
            out, S_state, z_state = oracle.oracle_fwd(q, k, v, om, C, ex["feature"])
            worst = max(worst, np.abs(out[0, 0] - np.array(ex["out"])).max(),
                        np.abs(S_state[0, 0] - np.array(ex["S_state"])).max(),
                        np.abs(z_state[0, 0] - np.array(ex["z_state"])).max())
            if "dv" in ex:
                dout = np.array(ex["dout"])[None, None]
                dq, dk, dv, _, _ = oracle.oracle_bwd(q, k, v, om, dout, S_state, z_state,
                                                     C, ex["feature"])
                worst = max(worst, np.abs(dv[0, 0] - np.array(ex["dv"])).max(),
                            np.abs(dq[0, 0] - np.array(ex["dq"])).max())
    return worst


def pin_autograd_brute(feature):
    """Library cross-check: torch.autograd (fp64, CPU) through the quadratic
    masked formula against the sliced backward sweep."""
    torch = pytest.importorskip("torch")
    Q, K, V, Omega, dY = small_case(13, chains=2, L=20, d=3, M=5, feature=feature)
    tQ, tK, tV, tO = (torch.tensor(a, requires_grad=True) for a in (Q, K, V, Omega))

    def g(X):
        if feature == "square":
            return X * X
        p = X @ tO.T
        if feature == "exp":
            return torch.exp(p - 0.5 * (X * X).sum(-1, keepdim=True)) / math.sqrt(tO.shape[0])
        return torch.relu(p) / math.sqrt(tO.shape[0])

    A = torch.tril(g(tQ) @ g(tK).transpose(1, 2))
    Y = (A @ tV) / A.sum(-1, keepdim=True)
    (Y * torch.tensor(dY)).sum().backward()
    _, R, S = sliced.forward(Q, K, V, Omega, 6, feature)
    dQ, dK, dV, dO, _, _ = sliced.backward(Q, K, V, Omega, dY, 6, feature, R, S)
    gO = tO.grad.numpy() if tO.grad is not None else np.zeros_like(Omega)
    if feature == "square":  # Omega is not used: its gradient is zero
        return max(rel(dQ, tQ.grad.numpy()), rel(dK, tK.grad.numpy()),
                   rel(dV, tV.grad.numpy()), float(np.abs(dO).max()), float(np.abs(gO).max()))
    return max(rel(dQ, tQ.grad.numpy()), rel(dK, tK.grad.numpy()),
               rel(dV, tV.grad.numpy()), rel(dO, gO))


# ----------------------------------------------------------------------------- tests

@pytest.mark.parametrize("feature", ["exp", "relu", "square"])
def test_brute_vs_sliced(feature):
    assert pin_brute_vs_sliced(feature) < 1e-12


def test_zero_omega_closed_form():
    assert pin_zero_omega_closed_form() < 1e-13


@pytest.mark.parametrize("feature", ["exp", "relu", "square"])
def test_final_state_closed_form(feature):
    assert pin_final_state_closed_form(feature) < 1e-13


@pytest.mark.parametrize("feature", ["exp", "relu", "square"])
def test_recurrence_forward(feature):
    assert pin_recurrence_forward(feature) < 1e-12


@pytest.mark.parametrize("feature", ["exp", "relu", "square"])
def test_recurrence_backward(feature):
    assert pin_recurrence_backward(feature) < 1e-11


@pytest.mark.parametrize("feature", ["exp", "relu", "square"])
def test_finite_differences(feature):
    assert pin_finite_differences(feature) < 1e-6


@pytest.mark.parametrize("feature", ["exp", "relu", "square"])
def test_rollback_closes(feature):
    assert pin_rollback_closes(feature) < 1e-12


def test_initial_state_gradient():
    assert pin_initial_state_gradient() < 1e-7


@pytest.mark.parametrize("feature", ["exp", "relu", "square"])
def test_streaming_continuation(feature):
    assert pin_streaming_continuation(feature) < 1e-12


def test_favor_unbiased():
    assert pin_favor_unbiased() < 0.03


def test_relu_arccos_kernel():
    assert pin_relu_arccos() < 0.03


@pytest.mark.parametrize("feature", ["exp", "relu", "square"])
def test_block_equals_whole(feature):
    assert pin_block_equals_whole(feature) < 1e-12


def test_golden_hand_examples():
    assert pin_golden() < 1e-12


@pytest.mark.parametrize("feature", ["exp", "relu", "square"])
def test_autograd_cross_check(feature):
    assert pin_autograd_brute(feature) < 1e-10


def test_first_row_and_linearity():
    """Y_1 = V_1 (a single term in eq. 2); Y is linear in V; scaling the ReLU
    map's Omega by c > 0 scales g by c and cancels in the ratio."""
    Q, K, V, Omega, _ = small_case(14, feature="relu")
    V2 = np.random.default_rng(15).standard_normal(V.shape)
    f = lambda V_, Om: sliced.forward(Q, K, V_, Om, 5, "relu")[0]
    Y = f(V, Omega)
    assert np.allclose(Y[:, 0], V[:, 0], rtol=0, atol=1e-15)
    assert rel(f(V + 2 * V2, Omega), Y + 2 * f(V2, Omega)) < 1e-12
    assert rel(f(V, 3.0 * Omega), Y) < 1e-12


def test_slices_partition():
    """N = ceil(L/C), A_n = (n-1)C, B_n = C except a shorter last slice."""
    assert sliced.slices(10, 4) == [(0, 4), (4, 8), (8, 10)]
    assert sliced.slices(8, 4) == [(0, 4), (4, 8)]
    assert sliced.slices(5, 9) == [(0, 5)]
    assert sliced.slices(3, 1) == [(0, 1), (1, 2), (2, 3)]
    with pytest.raises(ValueError):
        sliced.slices(4, 0)


def test_relu_zero_denominator_rows():
    """A query with g(q) = 0 has an all-zero weight row: the oracle returns 0
    for that row and passes no gradient through it."""
    Q, K, V, Omega, dY = small_case(16, chains=1, L=6, feature="relu")
    Q[0, 3] = -Omega.sum(axis=0) * 1e3     # large negative projection on most rows
    Omega = np.abs(Omega)
    Q[0, 3] = -np.abs(Q[0, 3])              # omega_m . q < 0 for every m
    Y, R, S = sliced.forward(Q, K, V, Omega, 2, "relu")
    assert np.all(Y[0, 3] == 0.0)
    dQ, dK, dV, dO, _, _ = sliced.backward(Q, K, V, Omega, dY, 2, "relu", R, S)
    assert np.all(np.isfinite(dQ)) and np.all(dQ[0, 3] == 0.0)


def pin_square_map_closed_form():
    """The quadratic map (Sec. 4): g(q).g(k) = sum_i q_i^2 k_i^2, so with every
    key equal to e_1 (g(k) = e_1) each weight is q_{l,1}^2 and the output is the
    plain causal mean of the values; and dOmega = 0 (no random features)."""
    rng = np.random.default_rng(17)
    L, d = 9, 3
    Q = rng.standard_normal((1, L, d)) + 2.0
    K = np.zeros((1, L, d))
    K[..., 0] = 1.0
    V = rng.standard_normal((1, L, d))
    Y, _, _ = sliced.forward(Q, K, V, np.zeros((d, d)), 4, "square")
    mean = np.cumsum(V[0], axis=0) / np.arange(1, L + 1)[:, None]
    return rel(Y[0], mean)


def test_square_map_closed_form():
    assert pin_square_map_closed_form() < 1e-13


def pin_streaming_backward(feature):
    """Two segments: the backward of the later segment hands its G^(0) to the
    backward of the earlier one as G^(N) (Sec. 3.3: G^(n) is the gradient with
    respect to the state a segment starts from).  Gradients of the two calls
    together equal the gradients of one call over the whole sequence."""
    Q, K, V, Omega, dY = small_case(18, feature=feature)
    rng = np.random.default_rng(19)
    a, C = 23, 6
    q, k, v, do = (x[:, None] for x in (Q, K, V, dY))     # [B, H=1, L, d]
    o, S, z = oracle.oracle_fwd(q, k, v, Omega, C, feature)
    full = oracle.oracle_bwd(q, k, v, Omega, do, S, z, C, feature)
    _, S1, z1 = oracle.oracle_fwd(q[:, :, :a], k[:, :, :a], v[:, :, :a], Omega, C, feature)
    _, S2, z2 = oracle.oracle_fwd(q[:, :, a:], k[:, :, a:], v[:, :, a:], Omega, C, feature, S1, z1)
    late = oracle.oracle_bwd(q[:, :, a:], k[:, :, a:], v[:, :, a:], Omega, do[:, :, a:], S2, z2,
                             C, feature)
    early = oracle.oracle_bwd(q[:, :, :a], k[:, :, :a], v[:, :, :a], Omega, do[:, :, :a], S1, z1,
                              C, feature, late[4]["G_S"], late[4]["g_z"])
    errs = [rel(np.concatenate([early[i], late[i]], axis=2), full[i]) for i in range(3)]
    errs.append(float(np.abs(early[3] + late[3] - full[3]).max()
                      / max(np.abs(full[3]).max(), 1e-300)))
    errs.append(rel(early[4]["G_S"], full[4]["G_S"]))
    return max(errs)


@pytest.mark.parametrize("feature", ["exp", "relu", "square"])
def test_streaming_backward(feature):
    assert pin_streaming_backward(feature) < 1e-12


# ----------------------------------------------------------------------------- non-causal form

from oracle import bidir  # noqa: E402


def pin_bidir_quadratic_vs_sweeps(feature, Cs=(1, 3, 16, 40, 64)):
    """The non-causal definition row by row against the two slice sweeps, for
    several slice sizes (the result does not depend on C)."""
    Q, K, V, Omega, _ = small_case(20, feature=feature)
    Yq = bidir.quadratic(Q, K, V, Omega, feature)
    return max(rel(bidir.forward(Q, K, V, Omega, C, feature)[0], Yq) for C in Cs)


def pin_bidir_zero_omega_closed_form():
    """Omega = 0 with the exp map: every weight is w_j = exp(-|k_j|^2/2)/M,
    independent of the query, so every row is the same global weighted mean."""
    Q, K, V, _, _ = small_case(21, chains=1, L=30)
    Y, _, _ = bidir.forward(Q, K, V, np.zeros((5, Q.shape[-1])), 7, "exp")
    w = np.exp(-0.5 * np.sum(K[0] ** 2, axis=1))
    mean = (w[:, None] * V[0]).sum(axis=0) / w.sum()
    return rel(Y[0], np.broadcast_to(mean, Y[0].shape))


def pin_bidir_finite_differences(feature, C=3):
    """Central differences of <dY, Y> on the row-by-row definition against the
    two backward sweeps."""
    Q, K, V, Omega, dY = small_case(22, chains=1, L=7, d=3, M=5, feature=feature)
    _, R, S = bidir.forward(Q, K, V, Omega, C, feature)
    dQ, dK, dV, dO, _ = bidir.backward(Q, K, V, Omega, dY, C, feature, R, S)
    fQ, fK, fV, fO = fd.central_differences(Q, K, V, Omega, dY, feature, fn=bidir.quadratic)
    return max(rel(dQ, fQ), rel(dK, fK), rel(dV, fV), rel(dO, fO))


def pin_bidir_last_row_is_causal():
    """The last row reads every key in both forms: there the non-causal output
    equals the causal one (eq. 2 at l = L), and the global state equals the
    causal final state."""
    Q, K, V, Omega, _ = small_case(23, feature="exp")
    Yb, Rb, Sb = bidir.forward(Q, K, V, Omega, 8, "exp")
    Yc, Rc, Sc = sliced.forward(Q, K, V, Omega, 8, "exp")
    return max(rel(Yb[:, -1], Yc[:, -1]), rel(Rb, Rc), rel(Sb, Sc))


@pytest.mark.parametrize("feature", ["exp", "relu", "square"])
def test_bidir_quadratic_vs_sweeps(feature):
    assert pin_bidir_quadratic_vs_sweeps(feature) < 1e-12


def test_bidir_zero_omega_closed_form():
    assert pin_bidir_zero_omega_closed_form() < 1e-13


@pytest.mark.parametrize("feature", ["exp", "relu", "square"])
def test_bidir_finite_differences(feature):
    assert pin_bidir_finite_differences(feature) < 1e-6


def test_bidir_last_row_is_causal():
    assert pin_bidir_last_row_is_causal() < 1e-12


# ----------------------------------------------------------------------------- the layer stack

from oracle import stack  # noqa: E402


def _stack_case(seed, s=3, chains=2, L=30, d=4, M=6, feature="exp"):
    rng = np.random.default_rng(seed)
    if feature == "square":
        M = d
    X = rng.standard_normal((chains, L, d)) * (0.5 if feature != "relu" else 1.0)
    Oms = [rng.standard_normal((M, d)) for _ in range(s)]
    dY = rng.standard_normal((chains, L, d))
    return X, Oms, dY


def pin_stack_quadratic_vs_sliced(feature, Cs=(1, 4, 7, 30, 64)):
    """The stack layer by layer with the row-by-row definition of eq. 2 against
    Algorithm 1's slice-outer, layer-inner sweep (one state per layer)."""
    X, Oms, _ = _stack_case(24, feature=feature)
    Yq = stack.quadratic(X, Oms, feature)
    return max(rel(stack.forward(X, Oms, C, feature)[0], Yq) for C in Cs)


def pin_stack_finite_differences(feature, C=3):
    """Central differences of <dY, X^(s)> (the layer-by-layer definition) with
    respect to X^(0) and every Omega_r, against the stack's backward sweep."""
    X, Oms, dY = _stack_case(25, s=2, chains=1, L=6, d=3, M=4, feature=feature)
    Y, states = stack.forward(X, Oms, C, feature)
    dX, dOm, B0 = stack.backward(X, Oms, dY, C, feature, states)

    def f():
        return float(np.sum(dY * stack.quadratic(X, Oms, feature)))

    h, worst = 1e-6, 0.0
    for arr, got in [(X, dX)] + list(zip(Oms, dOm)):
        fd = np.zeros_like(arr)
        it = np.nditer(arr, flags=["multi_index"])
        for _ in it:
            i = it.multi_index
            keep = arr[i]
            arr[i] = keep + h
            fp = f()
            arr[i] = keep - h
            fm = f()
            arr[i] = keep
            fd[i] = (fp - fm) / (2 * h)
        worst = max(worst, rel(got, fd))
    return worst


def pin_stack_rollback_closes():
    """After the reverse sweep every layer's state is rolled back to zero."""
    X, Oms, dY = _stack_case(26)
    _, states = stack.forward(X, Oms, 7, "exp")
    _, _, B0 = stack.backward(X, Oms, dY, 7, "exp", states)
    return max(max(np.abs(R).max() / np.abs(Rn).max(), np.abs(S).max() / np.abs(Sn).max())
               for (R, S), (Rn, Sn) in zip(B0, states))


def pin_stack_one_layer():
    """s = 1 is one layer plus the residual: X^(1) = X + Att(u, u, u) with u
    the normalised rows."""
    X, Oms, _ = _stack_case(27, s=1)
    Y, _ = stack.forward(X, Oms, 5, "relu")
    U = stack.row_norm(X)
    Yl, _, _ = sliced.forward(U, U, U, Oms[0], 5, "relu")
    return rel(Y, X + Yl)


def pin_row_norm():
    """The row normalisation: every row of u has root-mean-square d^(-1/4)
    (up to eps), u is invariant to scaling the row, and its VJP against
    central differences."""
    rng = np.random.default_rng(28)
    X = rng.standard_normal((2, 5, 8)) * 3.0
    U = stack.row_norm(X)
    d = X.shape[-1]
    err = float(np.abs(np.sqrt(np.mean(U * U, axis=-1)) - d ** -0.25).max())
    err = max(err, rel(stack.row_norm(7.0 * X), U))
    g = rng.standard_normal(X.shape)
    got = stack.row_norm_vjp(X, g)
    fd = np.zeros_like(X)
    h = 1e-6
    it = np.nditer(X, flags=["multi_index"])
    for _ in it:
        i = it.multi_index
        keep = X[i]
        X[i] = keep + h
        fp = float(np.sum(g * stack.row_norm(X)))
        X[i] = keep - h
        fm = float(np.sum(g * stack.row_norm(X)))
        X[i] = keep
        fd[i] = (fp - fm) / (2 * h)
    # eps = 1e-6 moves the root-mean-square and the scale invariance by
    # about eps / mean(x^2), well under 1e-5 for rows of scale 3
    return max(err / 1e-5, rel(got, fd) / 1e-6)


def test_row_norm():
    assert pin_row_norm() < 1.0


@pytest.mark.parametrize("feature", ["exp", "relu", "square"])
def test_stack_quadratic_vs_sliced(feature):
    assert pin_stack_quadratic_vs_sliced(feature) < 1e-12


@pytest.mark.parametrize("feature", ["exp", "square"])
def test_stack_finite_differences(feature):
    assert pin_stack_finite_differences(feature) < 1e-6


def test_stack_rollback_closes():
    assert pin_stack_rollback_closes() < 1e-11


def test_stack_one_layer():
    assert pin_stack_one_layer() < 1e-14
