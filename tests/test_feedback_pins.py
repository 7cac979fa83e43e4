"""Pins of the runtime feedback of the oracle: exit threshold (Eq. 37) and dual
weights (Eq. 43), against closed forms and their stated properties."""
import numpy as np
import pytest

from oracle import oracle as O


def _tok(T, N=8):
    return dict(pJ=np.full(T, 0.9, np.float32), alive=np.ones(T, np.uint8),
                exit_layer=np.full(T, N, np.int16), xi_last=np.full(T, -1.0, np.float32),
                Dhat=np.zeros(T, np.float32), Dbar=np.full(T, 0.02, np.float32))


def _run(tok, **kw):
    args = dict(N=8, user_size=4, eta=0.1, p_min=0.6, kappa=0.05, delay_sum_ms=0.0, ref_slots=0.0,
                d_ref=10.0, omega_D=0.5)
    args.update(kw)
    return O.feedback(tok, **args)


def test_exit_threshold_one_step_closed_form():
    """p <- p + eta (xi_mean - p), with xi_mean over the user's exited tokens."""
    tok = _tok(8)
    tok["alive"][[0, 2]] = 0
    tok["exit_layer"][[0, 2]] = 3
    tok["xi_last"][[0, 2]] = [0.96, 0.98]
    tok["xi_last"][1] = 0.5            # alive: not an exit, ignored
    pJ, out = _run(tok)
    want = np.float32(0.9) + np.float32(0.1) * (np.float32(0.97) - np.float32(0.9))
    assert pJ[:4] == pytest.approx(want, rel=1e-6)
    assert np.all(pJ[4:] == np.float32(0.9))          # user 1 had no exit
    assert out.users_updated == 1


def test_fixed_point_and_zero_step():
    tok = _tok(4)
    tok["alive"][:] = 0
    tok["exit_layer"][:] = 2
    tok["xi_last"][:] = 0.9
    pJ, _ = _run(tok)
    assert np.all(pJ == np.float32(0.9))
    tok["xi_last"][:] = 0.99
    pJ, _ = _run(tok, eta=0.0)
    assert np.all(pJ == np.float32(0.9))


def test_projection_onto_floor_and_one():
    tok = _tok(4)
    tok["alive"][:] = 0
    tok["exit_layer"][:] = 1
    tok["xi_last"][:] = 0.1
    pJ, _ = _run(tok, eta=0.9, p_min=0.75)
    assert np.all(pJ == np.float32(0.75))
    tok["xi_last"][:] = 1.0
    pJ, _ = _run(tok, eta=2.0)
    assert np.all(pJ == np.float32(1.0))


def test_exit_threshold_monotone_in_exit_confidence():
    prev = -1.0
    for x in np.linspace(0.6, 1.0, 9):
        tok = _tok(4)
        tok["alive"][0] = 0
        tok["exit_layer"][0] = 4
        tok["xi_last"][0] = x
        pJ, _ = _run(tok, p_min=0.0)
        assert pJ[0] >= prev
        prev = pJ[0]


def test_dual_weights_closed_form_and_bounds():
    # user 0: Dhat sums 0.02 of 0.08 -> 0.25; user 1: 0.04 of 0.08 -> 0.5; D_util = 0.375
    tok = _tok(8)
    tok["Dhat"][:4] = 0.005
    tok["Dhat"][4:] = 0.01
    # T_norm = 300 / (100 * 10) = 0.3
    pJ, out = _run(tok, delay_sum_ms=300.0, ref_slots=100.0, d_ref=10.0, kappa=0.2, omega_D=0.5)
    assert out.D_util == pytest.approx(0.375, rel=1e-6)
    assert out.T_norm == pytest.approx(0.3, rel=1e-12)
    assert out.omega_D == pytest.approx(0.5 + 0.2 * (0.375 - 0.3), rel=1e-6)
    assert out.omega_T == np.float32(1.0) - np.float32(out.omega_D)
    # utilisation above the delay raises omega_D; below lowers it; clipped to [0, 1]
    _, up = _run(tok, delay_sum_ms=0.0, ref_slots=100.0, kappa=10.0, omega_D=0.5)
    assert up.omega_D == 1.0 and up.omega_T == 0.0
    _, down = _run(tok, delay_sum_ms=1e6, ref_slots=100.0, kappa=10.0, omega_D=0.5)
    assert down.omega_D == 0.0 and down.omega_T == 1.0
