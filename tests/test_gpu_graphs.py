"""The forward replayed as a CUDA graph (trimmoe_config.graphs) gives exactly the
results of the plain launches, keeps the counters and records per-kernel
times through the events captured in the graph."""
import numpy as np
import pytest

from paper_2608_00573_gb300 import binding as B
from paper_2608_00573_gb300 import workload as W
from tests.gpu_helpers import make_engine
from tests.oracle_helpers import small_cfg

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="session", autouse=True)
def built_library():
    from paper_2608_00573_gb300 import build
    build.build()
    B.lib()


CASES = {
    "moe_shared_kc8": small_cfg(name="g1", N=4, d=256, E=16, k=4, F=128, F_sh=128, T=300, M=10, H=3,
                                n_centroids=8, seed=51),
    "full_block": small_cfg(name="g2", N=3, d=512, E=8, k=2, F=256, T=333, M=10, H=3, attn_heads=8,
                            attn_kv_heads=2, head_dim=64, attn_seq=128, seed=52),
    # K = 4096 down projections on both CTA-pair kernels draw their tiles from
    # per-layer counters, which every forward must start from zero
    "drawn_tiles": small_cfg(name="g3", N=3, d=512, E=4, k=2, F=4096, F_sh=4096, T=2100, M=10, H=3,
                             seed=53),
}


@pytest.mark.parametrize("name", list(CASES))
def test_graph_replay_equals_plain_launches(name):
    import torch
    cfg = CASES[name]
    plain, om, tables, small, experts = make_engine(cfg, theta=0.9, exit_bias=1.0)
    graph = B.Engine(cfg, tables, small, experts, T_max=cfg.T, profile=True, graphs=True)
    stream = torch.cuda.Stream()
    tok = W.make_tokens(cfg)
    with torch.cuda.stream(stream):
        pristine = plain.tokens_to_device(tok)
        buf_p = {k: v.clone() for k, v in pristine.items()}
        buf_g = {k: v.clone() for k, v in pristine.items()}
        # eager, capture + replay, then replays of both graph instances; the
        # counters restart before the third forward so that the graph engine's
        # kernel times come from the events inside the graph only
        for rep in range(5):
            if rep == 2:
                plain.reset_stats()
                graph.reset_stats()
            for k in pristine:
                buf_p[k].copy_(pristine[k])
                buf_g[k].copy_(pristine[k])
            plain.forward(buf_p, stream=stream)
            graph.forward(buf_g, stream=stream)
            stream.synchronize()
            a = B.Engine.tokens_to_host(buf_p)
            b = B.Engine.tokens_to_host(buf_g)
            if rep == 0:
                first = a
            for k in a:
                assert np.array_equal(a[k], b[k]), (rep, k)
                # the same inputs give the same forward every time
                assert np.array_equal(a[k], first[k]), (rep, k)
    sp, sg = plain.stats(), graph.stats()
    for key in ("layer_tokens", "exec_tokens", "skipped", "exited", "pairs_local_exact", "pairs_remote_sub",
                "launches", "layer_calls", "n_gemm_up", "n_gemm_down"):
        assert sp[key] == sg[key], key
    assert sg["gemm_flops"] == pytest.approx(sp["gemm_flops"])
    assert sg["flops_attn_gemm"] == pytest.approx(sp["flops_attn_gemm"])
    # per-kernel device time from the events inside the graph (3 replays)
    assert sg["ms_decide"] > 0 and sg["ms_gemm_up"] > 0 and sg["ms_router"] > 0
    assert sg["ms_gemm_up"] < 1e3
    assert sg["device_error"] == 0
    plain.close()
    graph.close()
    torch.cuda.synchronize()


def test_graph_dropped_when_tokens_move():
    """New token buffers (another key) run plainly first and match the plain
    engine again."""
    import torch
    cfg = CASES["moe_shared_kc8"]
    plain, om, tables, small, experts = make_engine(cfg, theta=0.9, exit_bias=1.0)
    graph = B.Engine(cfg, tables, small, experts, T_max=cfg.T, graphs=True)
    stream = torch.cuda.Stream()
    tok = W.make_tokens(cfg)
    with torch.cuda.stream(stream):
        pristine = plain.tokens_to_device(tok)
        for rep in range(4):
            buf_p = {k: v.clone() for k, v in pristine.items()}
            bufs = [{k: v.clone() for k, v in pristine.items()} for _ in range(2)]
            plain.forward(buf_p, stream=stream)
            for r2 in range(3):                     # same key three times: eager, graph, graph
                b = bufs[r2 % 2] if rep % 2 else bufs[0]
                for k in pristine:
                    b[k].copy_(pristine[k])
                graph.forward(b, stream=stream)
                stream.synchronize()
                x, y = B.Engine.tokens_to_host(buf_p), B.Engine.tokens_to_host(b)
                for k in x:
                    assert np.array_equal(x[k], y[k]), (rep, r2, k)
    plain.close()
    graph.close()
    torch.cuda.synchronize()


def test_graph_follows_feedback_updates():
    """Runtime feedback changes omega (a kernel parameter): the replayed graph
    is dropped and rebuilt, so forwards after the update equal those of plain
    launches with the same window sequence."""
    import torch
    cfg = CASES["moe_shared_kc8"]
    plain, om, tables, small, experts = make_engine(cfg, theta=0.9, exit_bias=1.0)
    graph = B.Engine(cfg, tables, small, experts, T_max=cfg.T, graphs=True)
    stream = torch.cuda.Stream()
    tok = W.make_tokens(cfg)
    with torch.cuda.stream(stream):
        pristine = plain.tokens_to_device(tok)
        buf_p = {k: v.clone() for k, v in pristine.items()}
        buf_g = {k: v.clone() for k, v in pristine.items()}
        for window in range(3):
            for rep in range(3):
                for k in pristine:
                    if k != "pJ":                       # p_J carries the feedback across windows
                        buf_p[k].copy_(pristine[k])
                        buf_g[k].copy_(pristine[k])
                plain.forward(buf_p, stream=stream)
                graph.forward(buf_g, stream=stream)
            op = plain.feedback(buf_p, user_size=128, eta=0.25, p_min=0.7, kappa=0.5, stream=stream)
            og = graph.feedback(buf_g, user_size=128, eta=0.25, p_min=0.7, kappa=0.5, stream=stream)
            assert op["omega_D"] == og["omega_D"] and op["omega_T"] == og["omega_T"], window
            stream.synchronize()
            a, b = B.Engine.tokens_to_host(buf_p), B.Engine.tokens_to_host(buf_g)
            for k in a:
                assert np.array_equal(a[k], b[k]), (window, k)
    plain.close()
    graph.close()
    torch.cuda.synchronize()
