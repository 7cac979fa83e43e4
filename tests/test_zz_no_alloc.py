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
from tests.gpu_helpers import make_engine
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
