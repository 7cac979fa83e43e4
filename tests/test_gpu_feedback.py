"""GPU parity of the runtime feedback (Eq. 37, 43) with the oracle, and of the
next forward that uses the updated weights and thresholds."""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2608_00573_gb300 import binding as B
from paper_2608_00573_gb300 import workload as W
from tests.gpu_helpers import compare_layer, make_engine
from tests.oracle_helpers import small_cfg

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("kappa", [0.05, 5.0])
def test_feedback_matches_oracle_and_next_forward_uses_it(kappa):
    import torch
    from paper_2608_00573_gb300 import build
    build.build()
    cfg = small_cfg(name="fb", N=4, d=256, E=8, k=2, F=256, T=640, M=10, H=3, seed=71)
    eng, om, tables, small, experts = make_engine(cfg, theta=0.9, exit_bias=1.0)
    dev = eng.tokens_to_device(W.make_tokens(cfg))
    eng.reset_stats()
    eng.forward(dev)
    torch.cuda.synchronize()
    before = B.Engine.tokens_to_host(dev)
    assert (before["alive"] == 0).sum() > 0
    out = eng.feedback(dev, user_size=128, eta=0.25, p_min=0.7, kappa=kappa)
    after = B.Engine.tokens_to_host(dev)
    assert out["window_ref_slots"] == cfg.T * cfg.k * cfg.N
    pJ_ref, o = O.feedback(before, cfg.N, 128, 0.25, 0.7, kappa, out["window_delay_ms"],
                           out["window_ref_slots"], tables["d_ref"], cfg.omega_D)
    assert np.array_equal(after["pJ"], pJ_ref)
    assert out["D_util"] == o.D_util and out["T_norm"] == o.T_norm
    assert out["omega_D"] == o.omega_D and out["omega_T"] == o.omega_T
    assert out["users_updated"] == o.users_updated > 0
    assert not np.array_equal(after["pJ"], before["pJ"])
    # next forward: new weights in the look-ahead and costs, new thresholds in the exit gate
    cfg2 = cfg.replace(omega_T=float(o.omega_T), omega_D=float(o.omega_D))
    om2 = O.OracleModel(cfg2, tables, small, experts)
    tok2 = W.make_tokens(cfg)
    tok2["pJ"] = after["pJ"]
    dev2 = eng.tokens_to_device(tok2)
    for l in range(cfg.N):
        compare_layer(cfg2, om2, eng, l, dev2, experts)
    eng.close()
