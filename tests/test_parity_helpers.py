"""The GPU parity checker's own logic, on the CPU.

The compaction check of tests/gpu_helpers.py rebuilds the expected order from
a layer's decisions; here it is run on oracle layers (with and without a
shared expert), must accept them, and must reject planted mistakes (two pairs
swapped inside a group, a pair moved across a group boundary, a shifted group
offset, a token whose decisions differ).  The targeted row selector must hit
the first and last row of every group and of every 128-row block.
"""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2608_00573_gb300 import workload as W
from tests.gpu_helpers import check_compaction, expected_compaction, targeted_rows
from tests.oracle_helpers import build_small, small_cfg


def _oracle_layers(cfg, theta=0.7, exit_bias=1.0):
    om, *_ = build_small(cfg, theta=theta, exit_bias=exit_bias)
    tok = W.make_tokens(cfg)
    h = tok.pop("h")
    outs = []
    for l in range(cfg.N):
        h, tok, out = O.layer_step(om, l, h, tok)
        outs.append(out)
    return outs


@pytest.mark.parametrize("F_sh", [0, 128])
def test_expected_compaction_equals_oracle(F_sh):
    cfg = small_cfg(k=2, T=300, N=3, F_sh=F_sh)
    for out in _oracle_layers(cfg):
        perm, goff = expected_compaction(out["action"], out["exp_sel"], cfg.T, cfg.k, cfg.E, F_sh > 0)
        assert np.array_equal(goff, out["group_off"])
        assert np.array_equal(perm, out["perm"][: int(goff[cfg.E + 1])])
        same = np.ones(cfg.T, bool)
        check_compaction(out, out, same, cfg.T, cfg.k, cfg.E, F_sh > 0, 0)


def test_compaction_check_rejects_planted_mistakes():
    cfg = small_cfg(k=2, T=300, N=2, F_sh=128)
    out = _oracle_layers(cfg)[1]
    T, K, E = cfg.T, cfg.k, cfg.E
    go = out["group_off"]
    same = np.ones(T, bool)
    big = int(np.argmax(np.diff(go[: E + 1])))
    a = int(go[big])

    def bad(mut):
        g = {k: np.array(v, copy=True) for k, v in out.items()}
        mut(g)
        with pytest.raises(AssertionError):
            check_compaction(g, out, same, T, K, E, True, 0)

    def swap(g):
        g["perm"][a], g["perm"][a + 1] = g["perm"][a + 1], g["perm"][a]
    bad(swap)

    def shift_offset(g):
        g["group_off"][big + 1] -= 1
    bad(shift_offset)

    def cross(g):
        b = int(go[big + 1])
        g["perm"][b - 1], g["perm"][b] = g["perm"][b], g["perm"][b - 1]
    if go[big + 1] < go[E]:
        bad(cross)

    # The GPU (here: a copy) executes a different expert for one token whose
    # decisions are counted as agreeing: its own stable sort still holds, so the
    # restricted comparison with the oracle must catch it.
    def other_expert(g):
        t = int(g["perm"][a]) // K
        j = int(g["perm"][a]) % K
        ex = g["exp_sel"].copy()
        ex[t * K + j] = (ex[t * K + j] + 1) % E
        perm, goff = expected_compaction(g["action"], ex, T, K, E, True)
        g["exp_sel"] = ex
        g["perm"][: len(perm)] = perm
        g["group_off"] = goff
    bad(other_expert)


def test_targeted_rows_cover_group_and_block_edges():
    T, K, E = 1000, 2, 4
    rng = np.random.default_rng(0)
    action = np.zeros(T, np.uint8)
    exp_sel = rng.integers(0, E, size=T * K).astype(np.uint8)
    perm, goff = expected_compaction(action, exp_sel, T, K, E, True)
    g = dict(perm=perm, group_off=goff, action=action)
    rows = set(targeted_rows(g, T, K, E, tiles=True).tolist())
    for e in range(E + 1):
        a, b = int(goff[e]), int(goff[e + 1])
        div = 1 if e == E else K
        for s in range(a, b, 128):
            assert int(perm[s]) // div in rows
            assert int(perm[min(s + 127, b - 1)]) // div in rows
    edges_only = set(targeted_rows(g, T, K, E).tolist())
    for e in range(E + 1):
        a, b = int(goff[e]), int(goff[e + 1])
        div = 1 if e == E else K
        assert int(perm[a]) // div in edges_only and int(perm[b - 1]) // div in edges_only
    assert edges_only <= rows
