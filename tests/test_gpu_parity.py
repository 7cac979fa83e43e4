"""GPU parity: the CUDA library (through the C ABI) against the CPU oracle.

Small configurations run every layer teacher-forced with every row checked;
the model-sized configurations check every decision and a seeded sample of
hidden rows at the sizes and launch configuration the benchmark uses.
"""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2608_00573_gb300 import binding as B
from paper_2608_00573_gb300 import workload as W
from tests.gpu_helpers import compare_layer, make_engine
from tests.oracle_helpers import small_cfg

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="session", autouse=True)
def built_library():
    from paper_2608_00573_gb300 import build
    build.build()
    B.lib()


def _run_all_layers(cfg, T=None, mutate_tokens=None, layers=None, row_sample=None, theta=None,
                    exit_bias=None):
    import torch
    eng, om, tables, small, experts = make_engine(cfg, T_max=T or cfg.T, theta=theta, exit_bias=exit_bias)
    tok = W.make_tokens(cfg, T=T)
    if mutate_tokens:
        mutate_tokens(tok)
    dev = eng.tokens_to_device(tok)
    reports = []
    for l in (layers if layers is not None else range(cfg.N)):
        reports.append(compare_layer(cfg, om, eng, l, dev, experts, row_sample=row_sample))
    eng.close()
    torch.cuda.synchronize()
    return reports


# (config, theta, exit-head bias): thresholds chosen so every action occurs.
SMALL = {
    "switch_tiny": W.CONFIGS["switch_tiny"],
    "swiglu_shared_k4": small_cfg(name="s1", N=3, d=512, E=16, k=4, F=384, F_sh=256, T=1000, M=10,
                                  H=3, zipf_s=0.8, seed=21),
    "swiglu_k2_renorm_h2": small_cfg(name="s2", N=4, d=256, E=8, k=2, F=256, T=333, M=10, H=2,
                                     renorm_topk=1, seed=22),
    "relu_k1_c64": small_cfg(name="s3", N=3, d=768, E=8, k=1, F=512, C=64, act=W.ACT_RELU, T=200,
                             M=10, seed=23),
    "e60_k4_h3": small_cfg(name="s4", N=4, d=256, E=60, k=4, F=128, F_sh=128, T=300, M=10, H=3,
                           zipf_s=1.0, seed=24),
    # ~300 rows per expert and K = F = 4096: the down projection runs on the
    # transposed pair kernel with tiles drawn from the launch-wide counter
    "dyn_tiles_f4096": small_cfg(name="s5", N=3, d=512, E=4, k=2, F=4096, T=600, M=10, H=3,
                                 zipf_s=0.5, seed=25),
    # 2100 live tokens through a shared expert of F_sh = 4096: its down
    # projection runs on the CTA-pair kernel with tiles drawn from the counter
    "shared_f4096_pair_dyn": small_cfg(name="s6", N=3, d=512, E=4, k=2, F=256, F_sh=4096, T=2100, M=10,
                                       H=3, zipf_s=0.5, seed=26),
}


KNOBS = {"switch_tiny": (None, None), "swiglu_shared_k4": (0.9, 1.0), "swiglu_k2_renorm_h2": (0.9, 1.0),
         "relu_k1_c64": (0.9, 5.0), "e60_k4_h3": (0.6, 1.0), "dyn_tiles_f4096": (0.9, 1.0),
         "shared_f4096_pair_dyn": (0.9, 1.0)}


@pytest.mark.parametrize("name", list(SMALL))
def test_layer_parity_small(name):
    cfg = SMALL[name]
    theta, bias = KNOBS[name]
    reports = _run_all_layers(cfg, theta=theta, exit_bias=bias)
    tot = {k: sum(r[k] for r in reports) for k in ("exec", "skip", "exit", "near_mismatch")}
    print(name, tot, [round(r["max_rel_err"], 5) for r in reports])
    assert tot["exec"] > 0
    if name != "switch_tiny":
        assert tot["skip"] > 0 and tot["exit"] > 0, tot


def test_tiny_free_running_forward_matches_oracle():
    """switch_tiny end to end without teacher forcing."""
    import torch
    cfg = W.CONFIGS["switch_tiny"]
    eng, om, tables, small, experts = make_engine(cfg)
    tok = W.make_tokens(cfg)
    dev = eng.tokens_to_device(tok)
    eng.forward(dev)
    torch.cuda.synchronize()
    got = B.Engine.tokens_to_host(dev)
    h0 = tok.pop("h")
    h_or, tok_or = O.forward(om, h0, tok)
    for k in ("s", "alive", "exit_layer", "last_exec"):
        assert np.array_equal(got[k], tok_or[k]), k
    # Without teacher forcing the hidden states drift by about one bf16 ulp per
    # layer, which moves the importance I (and a skip's Lambda = lambda * I) by
    # ~1e-5 of budget; decisions above are still required to match exactly.
    assert np.abs(got["Dhat"] - tok_or["Dhat"]).max() < 1e-4
    hg = W.bf16_bits_to_f32(got["h"]).astype(np.float64)
    ho = W.bf16_bits_to_f32(h_or).astype(np.float64)
    err = np.abs(hg - ho).max(axis=1) / np.abs(ho).max(axis=1)
    assert err.max() <= 2e-2
    eng.close()


def test_edge_cases_empty_single_and_dead():
    import torch
    cfg = SMALL["swiglu_shared_k4"]
    eng, om, tables, small, experts = make_engine(cfg, T_max=1000)
    # T = 0: a no-op
    tok = W.make_tokens(cfg, T=1000)
    dev = eng.tokens_to_device(tok)
    h_before = dev["hidden"].clone()
    eng.layer_step(0, dev, T=0)
    torch.cuda.synchronize()
    assert torch.equal(h_before, dev["hidden"])
    # T = 1
    tok1 = W.make_tokens(cfg, T=1)
    r = compare_layer(cfg, om, eng, 0, eng.tokens_to_device(tok1), experts)
    assert r["live"] == 1
    # all tokens dead: nothing changes
    tokd = W.make_tokens(cfg, T=257)
    tokd["alive"][:] = 0
    devd = eng.tokens_to_device(tokd)
    r = compare_layer(cfg, om, eng, 1, devd, experts)
    assert r["dead"] == 257
    # exited mid-way: every other token dead, layer > 0 with last_exec set
    tokh = W.make_tokens(cfg, T=999)
    tokh["alive"][::2] = 0
    tokh["last_exec"][:] = 1
    r = compare_layer(cfg, om, eng, 2, eng.tokens_to_device(tokh), experts)
    assert r["dead"] == 500
    eng.close()


@pytest.mark.parametrize("shared", [0, 256])
def test_all_tokens_skip(shared):
    """Every token sits on a server without any candidate, importance always
    under theta and a near-free skip: the whole layer is skipped."""
    cfg = small_cfg(name="skipall", N=2, d=256, E=8, k=2, F=256, F_sh=shared, T=300, M=4, H=1,
                    n_sub=0, seed=31)
    import torch
    small = W.make_small_weights(cfg)
    tables = W.make_tables(cfg, small["W_r"])
    tables["place"][:] = np.uint16(0b1110)          # nothing on server 0
    tables["theta"][:] = 1.0
    tables["lam"][:] = 1e-6
    experts = W.make_expert_weights_host(cfg)
    eng = B.Engine(cfg, tables, small, experts, T_max=cfg.T)
    om = O.OracleModel(cfg, tables, small, experts)
    tok = W.make_tokens(cfg)
    tok["s"][:] = 0
    r = compare_layer(cfg, om, eng, 0, eng.tokens_to_device(tok), experts)
    assert r["skip"] == cfg.T
    eng.close()
    torch.cuda.synchronize()


def test_empty_experts_and_concentrated_routing():
    """Strong router bias: most experts receive no pair (empty groups in the GEMM)."""
    cfg = small_cfg(name="skew", N=2, d=256, E=16, k=2, F=256, T=500, M=10, zipf_s=6.0, seed=41)
    reports = _run_all_layers(cfg)
    assert all(r["exec"] > 0 for r in reports)


def test_forward_host_equals_device_forward():
    import torch
    cfg = SMALL["swiglu_shared_k4"]
    eng, om, tables, small, experts = make_engine(cfg, T_max=1000)
    tok = W.make_tokens(cfg, T=1000)
    dev = eng.tokens_to_device(tok)
    eng.forward(dev)
    torch.cuda.synchronize()
    want = B.Engine.tokens_to_host(dev)
    host = {k: v.cpu().pin_memory() for k, v in eng.tokens_to_device(tok).items()}
    eng.forward_host(host)
    got = B.Engine.tokens_to_host(host)
    for k in want:
        assert np.array_equal(want[k], got[k]), k
    st = eng.stats()
    assert st["status"] == 0 and st["device_error"] == 0
    assert st["exec_tokens"] + st["skipped"] + st["exited"] == st["layer_tokens"]
    eng.close()


def test_stats_counters_consistent():
    import torch
    cfg = SMALL["swiglu_k2_renorm_h2"]
    eng, om, tables, small, experts = make_engine(cfg, profile=True)
    tok = W.make_tokens(cfg)
    dev = eng.tokens_to_device(tok)
    eng.reset_stats()
    eng.forward(dev)
    st = eng.stats()
    assert st["status"] == 0
    pairs = st["pairs_local_exact"] + st["pairs_local_sub"] + st["pairs_remote_exact"] + st["pairs_remote_sub"]
    assert pairs == st["exec_tokens"] * cfg.k
    assert st["exec_tokens"] + st["skipped"] + st["exited"] == st["layer_tokens"]
    assert st["max_budget_ratio"] <= 1.0
    assert st["layer_calls"] == cfg.N and st["ms_gemm_up"] > 0
    host = B.Engine.tokens_to_host(dev)
    assert int((host["alive"] == 0).sum()) == st["exited"]
    eng.close()


def test_device_wait_timeout_is_reported_and_context_survives():
    """Failure detection without a fault: a bounded mbarrier wait that nothing
    completes runs out, the host reads DEVICE_TIMEOUT and the self-test code,
    the second warp (two-second limit) returns on the abort flag, a reset clears
    the flag, and the next layer step on the same context still matches the
    oracle."""
    import time
    import torch
    cfg = SMALL["swiglu_k2_renorm_h2"]
    eng, om, tables, small, experts = make_engine(cfg)
    dev = eng.tokens_to_device(W.make_tokens(cfg))
    compare_layer(cfg, om, eng, 0, dev, experts)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    rc = B.trimmoe_watchdog_selftest(eng.handle, 20000, eng.stream_ptr())
    wall = time.perf_counter() - t0
    assert rc == -6, (rc, B.trimmoe_last_error(eng.handle))
    assert 0.02 <= wall < 1.0, wall
    assert "ran out (code 6)" in B.trimmoe_last_error(eng.handle)
    st = eng.stats()
    assert st["status"] == -6 and st["device_error"] == 6
    eng.reset_stats()
    st = eng.stats()
    assert st["status"] == 0 and st["device_error"] == 0
    compare_layer(cfg, om, eng, 1, dev, experts)
    assert B.trimmoe_watchdog_selftest(eng.handle, 0, eng.stream_ptr()) == -1
    assert eng.stats()["device_error"] == 0
    eng.close()


def test_create_out_of_memory_returns_status_and_recovers():
    """Workspaces for 100 million tokens (terabytes) cannot be allocated:
    trimmoe_create returns ERR_OOM with a message, frees what it had already
    allocated, and a create that fits works afterwards on the same device."""
    import torch
    cfg = small_cfg(name="oom", N=2, d=4096, E=8, k=2, F=256, T=64, M=6, H=2, seed=71)
    small = W.make_small_weights(cfg)
    tables = W.make_tables(cfg, small["W_r"])
    experts = W.make_expert_weights_host(cfg)
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    with pytest.raises(B.TrimmoeError) as ei:
        B.Engine(cfg, tables, small, experts, T_max=100_000_000)
    assert ei.value.status == -3 and "allocation" in str(ei.value)
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] >= free0 - (512 << 20)
    eng = B.Engine(cfg, tables, small, experts, T_max=64)
    dev = eng.tokens_to_device(W.make_tokens(cfg))
    eng.layer_step(0, dev)
    torch.cuda.synchronize()
    assert eng.stats()["status"] == 0
    eng.close()


def test_create_rejects_bad_input():
    cfg = SMALL["swiglu_k2_renorm_h2"]
    small = W.make_small_weights(cfg)
    tables = W.make_tables(cfg, small["W_r"])
    experts = W.make_expert_weights_host(cfg)
    bad = dict(tables)
    bad["place"] = tables["place"].copy()
    bad["place"][1, 3] = 0
    with pytest.raises(B.TrimmoeError) as ei:
        B.Engine(cfg, bad, small, experts, T_max=16)
    assert ei.value.status == -5
    with pytest.raises(B.TrimmoeError) as ei:
        B.Engine(cfg.replace(d=200), tables, small, experts, T_max=16)
    assert ei.value.status == -2
    bad = dict(tables)
    bad["P"] = tables["P"] * 2
    with pytest.raises(B.TrimmoeError) as ei:
        B.Engine(cfg, bad, small, experts, T_max=16)
    assert ei.value.status == -1
    eng = B.Engine(cfg, tables, small, experts, T_max=16)
    tok = eng.tokens_to_device(W.make_tokens(cfg, T=16))
    with pytest.raises(B.TrimmoeError):
        eng.layer_step(cfg.N, tok)
    with pytest.raises(B.TrimmoeError):
        eng.layer_step(0, tok, T=17)
    eng.close()


@pytest.mark.parametrize("name,kw", [
    ("E128_k8_C256_H6", dict(N=4, d=256, E=128, k=8, F=128, C=256, M=8, H=6, T=300, zipf_s=0.5)),
    ("M16_E64_k8_shared", dict(N=3, d=512, E=64, k=8, F=256, F_sh=128, M=16, H=3, T=257)),
])
def test_layer_parity_at_maximum_dimensions(name, kw):
    """The largest E, k, M, C and H the library accepts (E <= 128, k <= 8, M <= 16,
    C <= 256, H <= 6, M*E <= 1024)."""
    cfg = small_cfg(name=name, seed=91, **kw)
    reports = _run_all_layers(cfg, theta=0.95, exit_bias=1.0 if cfg.C == 1 else 8.0)
    tot = {k: sum(r[k] for r in reports) for k in ("exec", "skip", "exit")}
    print(name, tot)
    assert tot["exec"] > 0


@pytest.mark.parametrize("name,kw", [
    ("swiglu_shared_k2", dict(N=2, d=256, E=4, k=2, F=384, F_sh=256, T=4500, M=10, H=3)),
    ("relu_k1_c64", dict(N=2, d=512, E=2, k=1, F=512, C=64, act=W.ACT_RELU, T=4400, M=10)),
])
def test_layer_parity_pair_gemm(name, kw):
    """Groups averaging >= 2048 rows (and the shared expert's T rows) run the
    grouped GEMM on CTA pairs (256-row tiles, tcgen05 cta_group::2); ragged
    group tails leave the odd CTA's rows partly or wholly past the group."""
    cfg = small_cfg(name=name, seed=98, **kw)
    reports = _run_all_layers(cfg, theta=0.9, exit_bias=1.0 if cfg.C == 1 else 5.0)
    tot = {k: sum(r[k] for r in reports) for k in ("exec", "skip", "exit")}
    print(name, tot, [round(r["max_rel_err"], 5) for r in reports])
    assert tot["exec"] > 0


@pytest.mark.parametrize("name,kw", [
    ("swiglu_E16_k2", dict(N=2, d=512, E=16, k=2, F=384, T=2300, M=10, H=3, zipf_s=1.0)),
    ("relu_E8_k1", dict(N=2, d=768, E=8, k=1, F=512, C=64, act=W.ACT_RELU, T=2300, M=10, zipf_s=1.0)),
])
def test_layer_parity_transposed_pair_gemm(name, kw):
    """Groups averaging >= 256 rows run the routed down projection (and the
    ReLU up projection) on the transposed CTA-pair kernel: weights on the MMA's
    M side, a group's tokens on its N side in tiles of up to 256 rounded up to
    16.  With Zipf(1.0) routing the groups range from a few rows to well over
    256, so token tiles of many sizes (N from 16 to 256, tails inside a
    16-row step) occur."""
    cfg = small_cfg(name=name, seed=99, **kw)
    reports = _run_all_layers(cfg, theta=0.9, exit_bias=1.0 if cfg.C == 1 else 5.0)
    tot = {k: sum(r[k] for r in reports) for k in ("exec", "skip", "exit")}
    print(name, tot, [round(r["max_rel_err"], 5) for r in reports])
    assert tot["exec"] > 0


def test_layer_parity_decision_lane_groups_of_16():
    """8 < E <= 16 with more tokens than the resident warps (T >= 16 x SMs):
    the decision kernel runs two tokens per warp on 16-lane groups."""
    cfg = small_cfg(name="g16", N=2, d=256, E=16, k=2, F=128, T=2600, M=10, H=3, seed=99)
    reports = _run_all_layers(cfg, theta=0.9, exit_bias=1.0, row_sample=np.arange(0, 2600, 5))
    tot = {k: sum(r[k] for r in reports) for k in ("exec", "skip", "exit")}
    print("g16", tot)
    assert tot["exec"] > 0 and tot["skip"] > 0 and tot["exit"] > 0, tot


@pytest.mark.parametrize("budget", [0.0, float("inf")])
def test_budget_edge_cases(budget):
    """Dbar = 0: only exact execution fits (Q = 0), no skip; Dbar = inf: every
    substitute and skip fits and Q / Dbar = 0."""
    cfg = small_cfg(name="budget", N=3, d=256, E=8, k=2, F=256, T=300, M=10, seed=93)
    def mut(tok):
        tok["Dbar"][:] = budget
    reports = _run_all_layers(cfg, mutate_tokens=mut, theta=0.95, exit_bias=1.0)
    if budget == 0.0:
        assert sum(r["skip"] for r in reports) == 0


@pytest.mark.parametrize("name,kw", [
    ("mixtral_like_kc64", dict(N=6, d=512, E=8, k=2, F=256, T=700, M=10, H=3, n_centroids=64, renorm_topk=1,
                               exit_peak=3.0)),
    ("qwen_like_kc32_shared", dict(N=4, d=256, E=60, k=4, F=128, F_sh=128, T=300, M=10, H=3, n_centroids=32)),
])
def test_layer_parity_with_exit_prediction(name, kw):
    """Token-similarity exit prediction (Eq. 36) on: the predicted exit layer is
    compared per token and the capped look-ahead through the decisions."""
    import torch
    cfg = small_cfg(name=name, seed=95, **kw)
    eng, om, tables, small, experts = make_engine(cfg, theta=0.9, exit_bias=1.0)
    dev = eng.tokens_to_device(W.make_tokens(cfg))
    capped = 0
    for l in range(cfg.N):
        compare_layer(cfg, om, eng, l, dev, experts)
        # tokens whose predicted exit shortens this layer's look-ahead (checked above)
        capped += int((np.floor(small["centroid_exit"][l] + 0.5) < l + cfg.H).sum())
    assert capped > 0
    eng.close()
    torch.cuda.synchronize()


@pytest.mark.parametrize("n_centroids,T", [(0, 4096), (32, 4096), (0, 64), (32, 1)])
def test_forward_tables_for_all_layers_equal_per_layer_tables(n_centroids, T):
    """trimmoe_forward builds every layer's shared look-ahead tables in one
    launch before the first layer and its decisions read them at any T;
    trimmoe_layer_step builds its layer's tables itself when the tokens
    outnumber them, and otherwise every token computes its own table.  Same
    values, same order of operations: the paths must agree bit for bit on
    every token's state and hidden row."""
    import torch
    cfg = small_cfg(name=f"all_tabs_{n_centroids}", N=5, d=256, E=60, k=4, F=128, F_sh=128, T=4096, M=10,
                    H=3, zipf_s=1.0, seed=96, n_centroids=n_centroids)
    eng, om, tables, small, experts = make_engine(cfg, theta=0.6, exit_bias=1.0)
    tok = W.make_tokens(cfg, T=T)
    a = eng.tokens_to_device(tok)
    b = eng.tokens_to_device(tok)
    eng.reset_stats()
    eng.forward(a)
    torch.cuda.synchronize()
    st_fwd = eng.stats()
    eng.reset_stats()
    for l in range(cfg.N):
        eng.layer_step(l, b)
    torch.cuda.synchronize()
    st_step = eng.stats()
    ha, hb = B.Engine.tokens_to_host(a), B.Engine.tokens_to_host(b)
    for key in ha:
        assert np.array_equal(ha[key], hb[key]), key
    if T >= 1024:
        assert st_fwd["lookahead_shared"] == st_step["lookahead_shared"] > 0
        assert st_fwd["launches"] < st_step["launches"]
    else:
        assert st_step["lookahead_shared"] == 0
        if T >= 64:
            assert st_fwd["lookahead_shared"] > 0
    eng.close()


@pytest.mark.parametrize("n_centroids", [0, 32])
def test_shared_lookahead_tables_with_mixed_budgets(n_centroids):
    """Many tokens of one budget read the look-ahead table (Eq. 39) of their
    remaining-budget interval, computed once per layer; tokens of another budget
    compute their own.  Both must equal the oracle, which computes every table
    per token.  Remaining budgets are spread over the whole range, and with exit
    prediction the window is shortened for some tokens."""
    import torch
    cfg = small_cfg(name=f"shared_phi_{n_centroids}", N=4, d=256, E=60, k=4, F=128, F_sh=128, T=4096, M=10,
                    H=3, zipf_s=1.0, seed=97, n_centroids=n_centroids)
    eng, om, tables, small, experts = make_engine(cfg, theta=0.6, exit_bias=1.0)
    tok = W.make_tokens(cfg)
    rng = np.random.default_rng(7)
    odd = np.arange(cfg.T) % 2 == 1
    tok["Dbar"][odd] = np.float32(cfg.budget * 0.5)
    tok["Dhat"] = (tok["Dbar"] * rng.random(cfg.T).astype(np.float32) ** 3).astype(np.float32)
    dev = eng.tokens_to_device(tok)
    eng.reset_stats()
    sample = rng.choice(cfg.T, size=384, replace=False)
    for l in range(cfg.N):
        compare_layer(cfg, om, eng, l, dev, experts, row_sample=sample)
    st = eng.stats()
    print(n_centroids, st["lookahead_shared"], st["layer_tokens"])
    assert 0 < st["lookahead_shared"] < st["layer_tokens"]
    eng.close()
    torch.cuda.synchronize()
