"""Pins of the token-similarity exit prediction (Eq. 36) in the oracle.

The predicted exit layer is the rounded average exit layer of the nearest
centroid (cosine similarity); layers from it on are predicted not to run, so
the look-ahead of Eq. (39) stops before them.  A cap reduces the look-ahead to
a shorter horizon, which is checked against models built with that horizon.
"""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2608_00573_gb300 import workload as W
from tests.oracle_helpers import build_small, small_cfg


def test_nearest_centroid_by_cosine_and_rounding():
    cfg = small_cfg(d=256, n_centroids=16)
    om, tables, small, _ = build_small(cfg, with_experts=False)
    rng = np.random.default_rng(0)
    C = W.bf16_bits_to_f32(small["centroids"][0]).astype(np.float64)
    ex = np.linspace(1.0, 3.9, 16).astype(np.float32)
    for _ in range(50):
        h = W.f32_to_bf16_bits(rng.standard_normal(cfg.d).astype(np.float32))
        L, best, gap = O.predict_exit(om, small["centroids"][0], ex, h)
        hf = W.bf16_bits_to_f32(h).astype(np.float64)
        cos = C @ hf / np.linalg.norm(C, axis=1) / np.linalg.norm(hf)
        j = int(np.argmax(cos))
        assert L == int(np.floor(ex[j] + 0.5))
    # rounding of the average exit layer: halves go up (a model with one centroid)
    om1 = O.OracleModel(cfg.replace(n_centroids=1), tables, small)
    one = np.zeros((1, cfg.d), np.uint16)
    one[0] = W.f32_to_bf16_bits(np.ones(cfg.d, np.float32))
    h = one[0]
    for avg, want in [(2.5, 3), (2.49, 2), (3.0, 3), (1.51, 2)]:
        L, _, _ = O.predict_exit(om1, one, np.array([avg], np.float32), h)
        assert L == want


@pytest.mark.parametrize("l", [0, 1])
def test_capped_lookahead_equals_shorter_horizon(l):
    """cap = 0 gives Phi = 0 (the myopic H = 1 case), cap = 1 the H = 2 table,
    cap >= H - 1 the uncapped table."""
    cfg3 = small_cfg(E=5, M=4, N=5, H=3)
    om3, tables, small, _ = build_small(cfg3, with_experts=False)
    om2 = O.OracleModel(cfg3.replace(H=2), tables, small)
    for R, Dbar in [(0.02, 0.02), (0.005, 0.02)]:
        assert not O.lookahead_table_capped(om3, l, R, Dbar, 0).any()
        assert np.array_equal(O.lookahead_table_capped(om3, l, R, Dbar, 1), O.lookahead_table(om2, l, R, Dbar))
        assert np.array_equal(O.lookahead_table_capped(om3, l, R, Dbar, 5), O.lookahead_table(om3, l, R, Dbar))


def _run_layers(om, cfg, tok):
    h = tok.pop("h")
    outs = []
    for l in range(cfg.N):
        h, tok, out = O.layer_step(om, l, h, tok, row_mask=np.zeros(len(h), np.uint8))
        outs.append(out)
    return outs


def test_prediction_at_next_layer_is_myopic_and_at_depth_is_neutral():
    """Every centroid predicting an exit at l + 1 truncates the look-ahead to
    nothing: decisions equal those of H = 1.  Predicting exit at N changes
    nothing against the model without prediction."""
    base = small_cfg(E=6, M=6, N=4, k=2, T=96, H=3, seed=5)
    cfgp = base.replace(n_centroids=4)
    _, tables, small, _ = build_small(cfgp, theta=0.9, exit_bias=1.0, with_experts=False)
    tok = W.make_tokens(base)
    # exit at the next layer everywhere -> equals H = 1
    sm = dict(small)
    sm["centroid_exit"] = np.array([[l + 1] * 4 for l in range(base.N)], np.float32)
    got = _run_layers(O.OracleModel(cfgp, tables, sm), cfgp, {k: v.copy() for k, v in tok.items()})
    want = _run_layers(O.OracleModel(base.replace(H=1), tables, small), base, {k: v.copy() for k, v in tok.items()})
    for a, b in zip(got, want):
        for key in ("action", "exp_sel", "srv_sel"):
            assert np.array_equal(a[key], b[key])
    # exit predicted at full depth -> equals no prediction
    sm["centroid_exit"] = np.full((base.N, 4), base.N, np.float32)
    got = _run_layers(O.OracleModel(cfgp, tables, sm), cfgp, {k: v.copy() for k, v in tok.items()})
    want = _run_layers(O.OracleModel(base, tables, small), base, {k: v.copy() for k, v in tok.items()})
    for a, b in zip(got, want):
        for key in ("action", "exp_sel", "srv_sel", "tot_exec"):
            assert np.array_equal(a[key], b[key])


def test_guarantees_hold_with_exit_prediction():
    cfg = small_cfg(k=2, T=128, N=6, E=8, M=10, n_sub=1, n_centroids=8, seed=9)
    om, tables, small, _ = build_small(cfg, theta=0.9, exit_bias=1.0, with_experts=False)
    tok = W.make_tokens(cfg)
    h = tok.pop("h")
    for l in range(cfg.N):
        before = {k: v.copy() for k, v in tok.items()}
        h, tok, out = O.layer_step(om, l, h, tok, row_mask=np.zeros(cfg.T, np.uint8))
        assert np.all(tok["Dhat"] <= tok["Dbar"])
        ex = out["action"] == O.A_EXIT
        assert np.all(out["xi"][ex] >= before["pJ"][ex])
