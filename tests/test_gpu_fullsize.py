"""GPU parity at the model-shaped sizes, in the launch configuration bench.py times.

Every decision of every token is compared with the oracle (teacher-forced per
layer); hidden states are compared on a seeded sample of rows, which the
oracle computes one by one.  Layers that are not checked still run on the GPU
so that later checked layers see realistic state (skips, exits, budgets).
"""
import numpy as np
import pytest

from paper_2608_00573_gb300 import workload as W
from tests.gpu_helpers import compare_layer, make_engine

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


@pytest.fixture(scope="module", autouse=True)
def built_library():
    from paper_2608_00573_gb300 import binding as B
    from paper_2608_00573_gb300 import build
    build.build()
    B.lib()


def _sample_rows(T, n, seed):
    rng = np.random.default_rng(seed)
    return np.sort(rng.choice(T, size=min(n, T), replace=False))


def _check(cfg, eng, om, experts, tok, check_layers, n_rows, T=None):
    import torch
    dev = eng.tokens_to_device(tok)
    T = dev["s"].shape[0]
    reports = []
    for l in range(cfg.N):
        if l in check_layers:
            r = compare_layer(cfg, om, eng, l, dev, experts, row_sample=_sample_rows(T, n_rows, 1000 + l))
            reports.append(r)
            print(cfg.name, T, r)
        else:
            eng.layer_step(l, dev)
    torch.cuda.synchronize()
    return reports


def test_switch_full_size():
    cfg = W.CONFIGS["switch"]
    eng, om, tables, small, experts = make_engine(cfg, device_experts=True)
    reps = _check(cfg, eng, om, experts, W.make_tokens(cfg), set(range(cfg.N)), 256)
    assert sum(r["skip"] for r in reps) > 0 and sum(r["exit"] for r in reps) > 0
    eng.close()


def test_qwen_full_size():
    cfg = W.CONFIGS["qwen"]
    eng, om, tables, small, experts = make_engine(cfg, device_experts=True)
    reps = _check(cfg, eng, om, experts, W.make_tokens(cfg), {0, 1, 12, 23}, 128)
    assert sum(r["skip"] for r in reps) > 0
    eng.close()


@pytest.fixture(scope="module")
def mixtral_experts():
    import torch
    ex = W.make_expert_weights_device(W.CONFIGS["mixtral"])
    yield ex
    del ex
    torch.cuda.empty_cache()


def test_mixtral_full_size(mixtral_experts):
    cfg = W.CONFIGS["mixtral"]
    eng, om, tables, small, experts = make_engine(cfg, experts=mixtral_experts)
    reps = _check(cfg, eng, om, experts, W.make_tokens(cfg), {0, 1, 20, 31}, 48)
    assert sum(r["skip"] for r in reps) > 0
    eng.close()


@pytest.mark.parametrize("T,budget", [(1, 0.02), (8, 0.02), (64, 0.005), (64, 0.02), (64, 0.05), (256, 0.02)])
def test_mixtral_decode(mixtral_experts, T, budget):
    """Decode-stress shapes: small batches, Zipf(1.5) routing, heavy exits
    (the Mixtral-shaped expert weights are shared with the forward case)."""
    cfg = W.CONFIGS["mixtral_decode"].replace(budget=budget)
    eng, om, tables, small, experts = make_engine(cfg, T_max=256, experts=mixtral_experts)
    tok = W.make_tokens(cfg, T=T, seed_offset=T)
    check = set(range(cfg.N)) if T <= 8 else {0, 12, 24, 31}
    _check(cfg, eng, om, experts, tok, check, 16)
    eng.close()
