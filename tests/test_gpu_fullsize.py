"""GPU parity at the model-shaped sizes, in the launch configuration bench.py times.

Every decision of every token is compared with the oracle (teacher-forced per
layer) and the compaction is checked bit for bit on every checked layer.
Hidden rows, which the oracle computes one by one, are chosen from the GPU's
compacted order: the first and last row of every expert group and of the
shared-expert rows, the odd CTA's first row in each group's ragged last tile,
plus seeded random rows; on one layer per workload also the first and last row
of every 128-row block of every group, so that every tile of both CTAs of
every grouped GEMM launch of that layer (including its last persistent round)
contributes a checked row.  Layers that are not checked still run on the GPU
so that later checked layers see realistic state (skips, exits, budgets).
"""
import pytest

from paper_2608_00573_gb300 import workload as W
from tests.gpu_helpers import compare_layer, make_engine, targeted_rows

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


@pytest.fixture(scope="module", autouse=True)
def built_library():
    from paper_2608_00573_gb300 import binding as B
    from paper_2608_00573_gb300 import build
    build.build()
    B.lib()


def _check(cfg, eng, om, experts, tok, check_layers, n_rows, tile_layers=()):
    import torch
    dev = eng.tokens_to_device(tok)
    T = dev["s"].shape[0]
    reports = []
    for l in range(cfg.N):
        if l in check_layers:
            def rows(g, l=l):
                return targeted_rows(g, T, cfg.k, cfg.E, tiles=l in tile_layers, extra=n_rows, seed=1000 + l)
            r = compare_layer(cfg, om, eng, l, dev, experts, row_sample=rows)
            reports.append(r)
            print(cfg.name, T, {k: v for k, v in r.items() if k not in ("oracle_out", "s_before")})
        else:
            eng.layer_step(l, dev)
    torch.cuda.synchronize()
    return reports


def test_switch_full_size():
    cfg = W.CONFIGS["switch"]
    eng, om, tables, small, experts = make_engine(cfg, device_experts=True)
    reps = _check(cfg, eng, om, experts, W.make_tokens(cfg), set(range(cfg.N)), 128, tile_layers=set(range(cfg.N)))
    assert sum(r["skip"] for r in reps) > 0 and sum(r["exit"] for r in reps) > 0
    eng.close()


def test_qwen_full_size():
    cfg = W.CONFIGS["qwen"]
    eng, om, tables, small, experts = make_engine(cfg, device_experts=True)
    reps = _check(cfg, eng, om, experts, W.make_tokens(cfg), {0, 1, 5, 9, 12, 16, 20, 23}, 64,
                  tile_layers={1})
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
    reps = _check(cfg, eng, om, experts, W.make_tokens(cfg), {0, 1, 4, 8, 12, 16, 20, 21, 24, 28, 31}, 32,
                  tile_layers={1})
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
    _check(cfg, eng, om, experts, tok, check, 16, tile_layers=check)
    eng.close()
