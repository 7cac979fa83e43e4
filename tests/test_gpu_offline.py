"""GPU parity of the offline-stage calibration counts (Algorithm 1, Eq. 26-28, 38):
counts accumulated by the decision kernel during a calibration forward equal
the oracle's counts from its own (teacher-forced) decisions."""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2608_00573_gb300 import workload as W
from tests.gpu_helpers import compare_layer, make_engine
from tests.oracle_helpers import small_cfg

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("k,E", [(2, 8), (4, 16)])
def test_calibration_counts_match_oracle(k, E):
    import torch
    from paper_2608_00573_gb300 import build
    build.build()
    cfg = small_cfg(name="calib", N=5, d=256, E=E, k=k, F=256, T=900, M=10, H=3, seed=81)
    eng, om, tables, small, experts = make_engine(cfg, theta=0.9, exit_bias=1.0)
    cc = O.CalibCounts(cfg)
    prev = np.full(cfg.T, -1, np.int16)
    eng.calibration_begin()
    dev = eng.tokens_to_device(W.make_tokens(cfg))
    for l in range(cfg.N):
        r = compare_layer(cfg, om, eng, l, dev, experts)
        assert r["near_mismatch"] == 0
        cc.accumulate(om, l, r["oracle_out"], r["s_before"], prev)
    got = eng.calibration_end(cfg.T)
    want = cc.finalize(om, cfg.T)
    for key in ("trans", "alive", "resid", "act", "above"):
        assert np.array_equal(got[key], getattr(cc, key)), key
    for key in ("P", "pi", "sigma", "rho"):
        assert np.array_equal(got[key], want[key]), key
    assert np.array_equal(got["act_freq"], want["act"]) and np.array_equal(got["lam"], want["lam"])
    # the derived tables feed a replication that keeps the deployment feasible
    size = np.full((cfg.N, cfg.E), 1.0)
    cap = np.full(cfg.M, float(cfg.N * cfg.E) / 2)
    place, added = O.replicate(om, got["lam"], got["rho"], size, cap * 0 + 1e9, tables["place"])
    assert np.all(place != 0)
    eng.close()
    torch.cuda.synchronize()
