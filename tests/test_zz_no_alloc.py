"""The allocation-free compaction entry point against the regular layer step.

trimmoe_compact_noalloc serves callers that cannot call cudaMalloc (for
example code running inside an allocator callback, or a process whose device
memory belongs entirely to another pool): its scratch is one static device
array, so it needs no handle and allocates nothing.  This file is collected
last so that a failure here never hides the other tests' results.
"""
import numpy as np
import pytest

from paper_2608_00573_gb300 import binding as B
from paper_2608_00573_gb300 import workload as W
from tests.gpu_helpers import expected_compaction, make_engine
from tests.oracle_helpers import small_cfg

pytestmark = pytest.mark.gpu


def test_compact_noalloc_matches_layer_step_on_consecutive_calls():
    import torch
    from paper_2608_00573_gb300 import build
    build.build()
    cfg = small_cfg(name="noalloc", N=3, d=256, E=16, k=4, F=256, F_sh=128, T=1000, M=10, H=2,
                    zipf_s=0.8, seed=61)
    eng, *_ = make_engine(cfg, theta=0.9, exit_bias=1.0)
    dev = eng.tokens_to_device(W.make_tokens(cfg))
    T, K, E = cfg.T, cfg.k, cfg.E
    stream = eng.stream_ptr()
    seen_skip = seen_exit = False
    for layer in range(2):                        # two calls in a row share the scratch
        out = eng.alloc_layer_out(T)
        eng.layer_step(layer, dev, out=out)
        perm = torch.full((T * K + T,), -7, dtype=torch.int32, device="cuda")
        goff = torch.full((E + 2,), -7, dtype=torch.int32, device="cuda")
        pos_pair = torch.full((T * K,), -7, dtype=torch.int32, device="cuda")
        pos_sh = torch.full((T,), -7, dtype=torch.int32, device="cuda")
        B.trimmoe_compact_noalloc(out["action"], out["exp_sel"], T, K, E, 1, perm, goff, pos_pair, pos_sh,
                                  stream)
        torch.cuda.synchronize()
        want_goff = out["group_off"].cpu().numpy()
        got_goff = goff.cpu().numpy()
        assert np.array_equal(got_goff, want_goff)
        n = int(want_goff[E + 1])
        assert np.array_equal(perm.cpu().numpy()[:n], out["perm"].cpu().numpy()[:n])
        act = out["action"].cpu().numpy()
        pp = pos_pair.cpu().numpy()
        pm = perm.cpu().numpy()
        ex = np.repeat(act == 0, K)
        assert np.all(pp[~ex] == -1)
        assert np.array_equal(pm[pp[ex]], np.nonzero(ex)[0])
        ps = pos_sh.cpu().numpy()
        sh = (act == 0) | (act == 1)
        assert np.array_equal(pm[want_goff[E] + ps[sh]], np.nonzero(sh)[0])
        assert np.all(ps[~sh] == -1)
        seen_skip |= bool((act == 1).any())
        seen_exit |= bool((act == 2).any())
    assert seen_skip and seen_exit
    eng.close()


def test_compact_noalloc_rejects_oversized_input():
    import torch
    a = torch.zeros(8, dtype=torch.uint8, device="cuda")
    i32 = torch.zeros(8, dtype=torch.int32, device="cuda")
    with pytest.raises(B.TrimmoeError) as ei:
        B.trimmoe_compact_noalloc(a, a, 65537, 1, 8, 0, i32, i32, i32, None)
    assert "65536" in str(ei.value)
    with pytest.raises(B.TrimmoeError):
        B.trimmoe_compact_noalloc(a, a, 8, 1, 129, 0, i32, i32, i32, None)


@pytest.mark.parametrize("has_shared", [0, 1])
@pytest.mark.parametrize("T", [0, 1, 200, 1000, 65536])
def test_compact_noalloc_matches_stable_sort_and_allocates_nothing(T, has_shared):
    """Synthetic decisions (all four actions, every expert) at the single-chunk
    size (T <= 256), several chunks, the 65536-token limit and T = 0: the
    output equals the stable sort by (expert, t, j) that defines the
    compaction, twice in a row, and after a first call the device's free
    memory does not change across a call."""
    import torch
    K, E = 2, 8
    rng = np.random.default_rng(T + 7 * has_shared)
    action_h = rng.choice(4, size=max(T, 1), p=[0.7, 0.15, 0.1, 0.05]).astype(np.uint8)[:T]
    exp_h = rng.integers(0, E, size=T * K).astype(np.uint8)
    exp_h[np.repeat(action_h != 0, K)] = 255          # as the layer step writes it
    action = torch.from_numpy(np.concatenate([action_h, np.zeros(1, np.uint8)])).cuda()
    exp_sel = torch.from_numpy(np.concatenate([exp_h, np.zeros(1, np.uint8)])).cuda()
    perm = torch.full((T * K + T + 1,), -7, dtype=torch.int32, device="cuda")
    goff = torch.full((E + 2,), -7, dtype=torch.int32, device="cuda")
    pos_pair = torch.full((T * K + 1,), -7, dtype=torch.int32, device="cuda")
    pos_sh = torch.full((T + 1,), -7, dtype=torch.int32, device="cuda") if has_shared else None
    stream = torch.cuda.current_stream().cuda_stream
    want_perm, want_goff = expected_compaction(action_h, exp_h, T, K, E, bool(has_shared))

    def call():
        B.trimmoe_compact_noalloc(action, exp_sel, T, K, E, has_shared, perm, goff, pos_pair, pos_sh, stream)
        torch.cuda.synchronize()

    call()                                           # first call: set-up on this device
    torch.cuda.synchronize()
    free_before = torch.cuda.mem_get_info()[0]
    for _ in range(2):
        perm.fill_(-7)
        call()
        assert np.array_equal(goff.cpu().numpy(), want_goff)
        got = perm.cpu().numpy()
        n = len(want_perm)
        assert np.array_equal(got[:n], want_perm)
        assert np.all(got[n:] == -7)                  # nothing written past the rows
        if T:
            pp = pos_pair.cpu().numpy()[:T * K]
            ex = np.repeat(action_h == 0, K)
            assert np.all(pp[~ex] == -1)
            assert np.array_equal(got[pp[ex]], np.nonzero(ex)[0])
    assert torch.cuda.mem_get_info()[0] == free_before
