"""Plant plausible mistakes in the oracle (on the CPU) and check that at least
one pin of tests/test_oracle_pins.py detects each of them."""
import numpy as np
import pytest

from oracle import features, sliced

import test_oracle_pins as P


def _exclusive_forward_rows(R, S, Qt, Kt, V):
    # mistake: exclusive mask (the query reads the state before its own key)
    T_S, T_R = sliced._T(Kt, V)
    U_S = S[:, None, :] + np.cumsum(T_S, axis=1) - T_S
    U_R = R[:, None, :, :] + np.cumsum(T_R, axis=1) - T_R
    Y, _ = sliced._readout(U_R, U_S, Qt)
    return Y, U_R[:, -1] + T_R[:, -1], U_S[:, -1] + T_S[:, -1]


def _g_exp_no_norm_term(X, Omega):
    # mistake: the -|x|^2/2 term dropped
    return np.exp(features.projection(X, Omega)) / np.sqrt(Omega.shape[0])


def _g_exp_no_scale(X, Omega):
    # mistake: 1/sqrt(M) dropped
    half_sq = 0.5 * np.sum(X * X, axis=-1, keepdims=True)
    return np.exp(features.projection(X, Omega) - half_sq)


def _vjp_no_norm_term(X, Omega, dG, feature):
    # mistake: exp map's -x sum(u) term dropped
    u = dG * features.g_exp(X, Omega)
    dX = np.einsum("...lm,md->...ld", u, Omega)
    return dX, u.reshape(-1, Omega.shape[0]).T @ X.reshape(-1, X.shape[-1])


def _wrap_backward_rows(mutate):
    orig = sliced._backward_rows

    def bad(R, S, G_R, G_S, Qt, Kt, V, dY):
        return mutate(orig, R, S, G_R, G_S, Qt, Kt, V, dY)
    return bad


def _drop_state_gradient(orig, R, S, G_R, G_S, Qt, Kt, V, dY):
    # mistake: G is not carried between slices (G^(n) treated as 0)
    return orig(R, S, 0 * G_R, 0 * G_S, Qt, Kt, V, dY)


def _rollback_wrong_sign(orig, R, S, G_R, G_S, Qt, Kt, V, dY):
    # mistake: eq. 17 with + instead of -
    T_S, T_R = sliced._T(Kt, V)
    out = list(orig(R + 2 * T_R.sum(1), S + 2 * T_S.sum(1), G_R, G_S, Qt, Kt, V, dY))
    return tuple(out)


def _drop_key_normaliser_share(orig, R, S, G_R, G_S, Qt, Kt, V, dY):
    # mistake: App. B's key gradient without the normaliser's share
    dQt, dKt, dV, R0, S0, G_R2, G_S2 = orig(R, S, G_R, G_S, Qt, Kt, V, dY)
    T_S, _ = sliced._T(Kt, V)
    # remove the suffix sum of dU_S from dKt
    U_S = S0[:, None, :] + np.cumsum(T_S, axis=1)
    _, den = sliced._readout(np.zeros(Qt.shape[:2] + (V.shape[-1], Qt.shape[-1])), U_S, Qt)
    Y = sliced._forward_rows(R0, S0, Qt, Kt, V)[0]
    dden = -np.sum(dY * Y, axis=-1) / den
    dU_S = dden[:, :, None] * Qt
    dU_S[:, -1] += G_S
    dT_S = np.flip(np.cumsum(np.flip(dU_S, axis=1), axis=1), axis=1)
    return dQt, dKt - dT_S, dV, R0, S0, G_R2, G_S2


def _square_vjp_missing_two(X, Omega, dG, feature):
    # mistake: quadratic map's derivative taken as x instead of 2x
    if feature != "square":
        return _orig_vjp(X, Omega, dG, feature)
    return X * dG, np.zeros_like(Omega)


def _g_abs(X, Omega):
    # mistake: |x| in place of x^2 for the quadratic map
    return np.abs(X)


_orig_vjp = features.feature_vjp


def _bidir_backward_drop_key_normaliser(Q, K, V, Omega, dY, C, feature, R, S):
    # mistake: the non-causal key gradient without the normaliser's share G_S
    from oracle import bidir
    orig = _BIDIR_BACKWARD
    dQ, dK, dV, dO, (G_R, G_S) = orig(Q, K, V, Omega, dY, C, feature, R, S)
    Kt = features.feature_map(K, Omega, feature)
    bad, _ = features.feature_vjp(K, Omega, np.broadcast_to(G_S[:, None, :], Kt.shape), feature)
    return dQ, dK - bad, dV, dO, (G_R, G_S)


from oracle import bidir as _bidir  # noqa: E402
_BIDIR_BACKWARD = _bidir.backward

from oracle import stack as _stack  # noqa: E402
_STACK_LAYER_BWD = _stack.layer_backward


def _stack_layer_bwd_drops_residual(Q, K, V, Omega, dY, C, feature, R, S, G_R, G_S):
    # mistake: the layer's gradient replaces dX instead of adding to it (the
    # residual path dropped); planted as a layer backward that cancels dY
    dq, dk, dv, dO, B0, G = _STACK_LAYER_BWD(Q, K, V, Omega, dY, C, feature, R, S, G_R, G_S)
    return dq - dY, dk, dv, dO, B0, G

_ROW_NORM_VJP = _stack.row_norm_vjp


def _row_norm_vjp_no_projection(X, g):
    # mistake: the normalisation's VJP as a plain rescale, without removing
    # the component along x
    d = X.shape[-1]
    r = np.sqrt(np.mean(X * X, axis=-1, keepdims=True) + _stack.EPS)
    return d ** -0.25 / r * g


MUTATIONS = {
    "exclusive_mask": (lambda mp: mp.setattr(sliced, "_forward_rows", _exclusive_forward_rows),
                       lambda: P.pin_brute_vs_sliced("exp"), 1e-6),
    "g_exp_missing_norm_term": (lambda mp: mp.setattr(features, "g_exp", _g_exp_no_norm_term),
                                lambda: P.pin_favor_unbiased(), 0.1),
    "g_exp_missing_scale": (lambda mp: mp.setattr(features, "g_exp", _g_exp_no_scale),
                            lambda: P.pin_favor_unbiased(), 0.1),
    "vjp_missing_norm_term": (lambda mp: mp.setattr(sliced, "feature_vjp", _vjp_no_norm_term),
                              lambda: P.pin_finite_differences("exp"), 1e-3),
    "state_gradient_not_carried": (
        lambda mp: mp.setattr(sliced, "_backward_rows", _wrap_backward_rows(_drop_state_gradient)),
        lambda: P.pin_finite_differences("exp"), 1e-3),
    "rollback_wrong_sign": (
        lambda mp: mp.setattr(sliced, "_backward_rows", _wrap_backward_rows(_rollback_wrong_sign)),
        lambda: P.pin_rollback_closes("exp"), 1e-3),
    "key_grad_missing_normaliser": (
        lambda mp: mp.setattr(sliced, "_backward_rows", _wrap_backward_rows(_drop_key_normaliser_share)),
        lambda: P.pin_finite_differences("exp"), 1e-3),
    "square_vjp_missing_factor_two": (
        lambda mp: mp.setattr(sliced, "feature_vjp", _square_vjp_missing_two),
        lambda: P.pin_finite_differences("square"), 1e-3),
    "square_map_is_abs": (lambda mp: mp.setattr(features, "g_square", _g_abs),
                          lambda: P.pin_golden(), 1e-6),
    "stack_residual_dropped": (
        lambda mp: mp.setattr(_stack, "layer_backward", _stack_layer_bwd_drops_residual),
        lambda: P.pin_stack_finite_differences("exp"), 1e-3),
    "stack_norm_vjp_no_projection": (
        lambda mp: mp.setattr(_stack, "row_norm_vjp", _row_norm_vjp_no_projection),
        lambda: P.pin_stack_finite_differences("exp"), 1e-3),
    "bidir_key_grad_missing_normaliser": (
        lambda mp: mp.setattr(_bidir, "backward", _bidir_backward_drop_key_normaliser),
        lambda: P.pin_bidir_finite_differences("exp"), 1e-3),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_mutation_is_caught(name, monkeypatch):
    plant, pin, threshold = MUTATIONS[name]
    plant(monkeypatch)
    err = pin()
    assert not (err < threshold), f"pin did not catch {name}: err={err}"
