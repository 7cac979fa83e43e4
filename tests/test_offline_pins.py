"""Pins of the offline stage (Algorithm 1) in the oracle: calibration statistics
(Eq. 26, 27, 38) and greedy communication-aware replication (Eq. 28, Property 1)."""
import itertools

import numpy as np
import pytest

from oracle import oracle as O
from tests.oracle_helpers import build_small, small_cfg


def _om(**kw):
    cfg = small_cfg(**kw)
    om, tables, small, _ = build_small(cfg, with_experts=False)
    return cfg, om, tables


def test_transition_and_activity_counts_by_hand():
    """4 tokens, 3 layers, top-1 over 3 experts; token 3 dies after layer 0."""
    cfg, om, tables = _om(N=3, E=3, k=1, M=4)
    theta = tables["theta"]
    routes = [[0, 1, 2, 0], [1, 1, 0, -1], [2, 2, 1, -1]]        # slot-0 target per layer and token
    I = [[0.9, 0.1, 0.9, 0.9], [0.1, 0.1, 0.9, 0.0], [0.9, 0.9, 0.1, 0.0]]
    s_before = [[0, 1, 1, 2], [0, 0, 3, 0], [1, 1, 1, 0]]
    cc = O.CalibCounts(cfg)
    prev = np.full(4, -1, np.int16)
    for l in range(3):
        act = np.array([0 if r >= 0 else 3 for r in routes[l]], np.uint8)
        out = dict(topk_idx=np.array([max(r, 0) for r in routes[l]], np.int32),
                   I=np.array(I[l], np.float32), action=act)
        cc.accumulate(om, l, out, np.array(s_before[l], np.uint8), prev)
    st = cc.finalize(om, 4)
    # transitions 0->1: tokens (0:0->1), (1:1->1), (2:2->0); 1->2: (0:1->2), (1:1->2), (2:0->1)
    want0 = np.zeros((3, 3)); want0[0, 1] = want0[1, 1] = want0[2, 0] = 1
    want1 = np.zeros((3, 3)); want1[1, 2] = 2; want1[0, 1] = 1
    assert np.array_equal(cc.trans[0], want0) and np.array_equal(cc.trans[1], want1)
    assert np.allclose(st["P"][1][1], [0, 0, 1]) and np.allclose(st["P"][1][2], [1 / 3] * 3)
    assert np.allclose(st["pi"], [1.0, 0.75, 0.75])
    assert list(cc.alive) == [4, 3, 3]
    # sigma: layer 0 expert 0 routed twice (tokens 0, 3), I = 0.9 both -> above theta iff theta < 0.9
    above = (np.array(I[0]) > theta[0])
    assert st["sigma"][0][0] == pytest.approx((int(above[0]) + int(above[3])) / 2)
    assert st["rho"][1][0] == pytest.approx(2 / 3)             # layer 1: tokens 0, 1 on server 0 of 3 live
    assert np.allclose(st["act"].sum(axis=1), 1.0)
    assert np.allclose(st["lam"], st["pi"][:, None] * st["sigma"] * st["act"])


def test_active_probability_is_non_increasing():
    """Eq. (26) with the monotone activity of Eq. (6)."""
    cfg, om, tables = _om(N=5, E=4, k=2, M=3)
    rng = np.random.default_rng(0)
    T = 200
    exit_at = rng.integers(1, 6, size=T)
    cc = O.CalibCounts(cfg)
    prev = np.full(T, -1, np.int16)
    for l in range(cfg.N):
        act = np.where(exit_at > l, 0, 3).astype(np.uint8)
        out = dict(topk_idx=rng.integers(0, 4, size=(T, 2)).astype(np.int32).ravel(),
                   I=rng.random(T).astype(np.float32), action=act)
        cc.accumulate(om, l, out, rng.integers(0, 3, size=T).astype(np.uint8), prev)
    pi = cc.finalize(om, T)["pi"]
    assert np.all(np.diff(pi) <= 0) and pi[0] == 1.0


def _random_replication_case(seed, N=3, E=4, M=4):
    cfg, om, tables = _om(N=N, E=E, M=M, k=1, seed=seed)
    rng = np.random.default_rng(seed)
    lam = rng.random((N, E)).astype(np.float32)
    rho = rng.dirichlet(np.ones(M), size=N).astype(np.float32)
    size = rng.integers(1, 4, size=(N, E)).astype(np.float64)
    place = np.zeros((N, E), np.uint16)
    for l in range(N):
        for e in range(E):
            place[l, e] = 1 << int(rng.integers(M))
    used = np.zeros(M)
    for l in range(N):
        for e in range(E):
            for m in range(M):
                if place[l, e] >> m & 1:
                    used[m] += size[l, e]
    cap = used + rng.integers(0, 8, size=M)
    return cfg, om, tables, lam, rho, size, cap, place


@pytest.mark.parametrize("seed", range(6))
def test_replication_keeps_deployment_feasible(seed):
    """Property 1: coverage (c.2) and memory (c.1) hold after Algorithm 1, and no
    feasible replica is left."""
    cfg, om, tables, lam, rho, size, cap, place = _random_replication_case(seed)
    new, added = O.replicate(om, lam, rho, size, cap, place)
    N, E, M = cfg.N, cfg.E, cfg.M
    assert np.all((new & place) == place)                  # replication only adds copies
    assert np.all(new != 0)
    used = np.zeros(M)
    for l in range(N):
        for e in range(E):
            for m in range(M):
                if new[l, e] >> m & 1:
                    used[m] += size[l, e]
    assert np.all(used <= cap)
    for l in range(N):
        for e in range(E):
            for m in range(M):
                if not new[l, e] >> m & 1:
                    assert used[m] + size[l, e] > cap[m]
    assert added == int(sum(bin(int(x)).count("1") for x in new.ravel()) - N * E)


@pytest.mark.parametrize("seed", range(6))
def test_replication_matches_bruteforce_greedy(seed):
    """Each step places the feasible pair of largest benefit (Eq. 28), ties to the
    lowest (m, l, k); enumerated independently here."""
    cfg, om, tables, lam, rho, size, cap, place = _random_replication_case(seed)
    trans = tables["trans"].astype(np.float64)
    N, E, M = cfg.N, cfg.E, cfg.M
    pl = place.copy()
    used = np.zeros(M)
    for l, e, m in itertools.product(range(N), range(E), range(M)):
        if pl[l, e] >> m & 1:
            used[m] += size[l, e]
    while True:
        cands = []
        for m, l, e in itertools.product(range(M), range(N), range(E)):
            if pl[l, e] >> m & 1 or used[m] + size[l, e] > cap[m]:
                continue
            hosts = [mp for mp in range(M) if pl[l, e] >> mp & 1]
            B = float(lam[l, e]) * float(rho[l, m]) * float(np.mean([trans[m, mp] for mp in hosts]))
            cands.append((-B, m, l, e))
        if not cands:
            break
        _, m, l, e = min(cands)
        pl[l, e] |= 1 << m
        used[m] += size[l, e]
    new, _ = O.replicate(om, lam, rho, size, cap, place)
    assert np.array_equal(new, pl)


def test_replication_benefit_by_hand():
    """Two servers, one layer, two experts on server 0 only.  trans[1][0] = d.
    Benefits on server 1: lambda_k * rho_{1} * d; memory for one replica only:
    the expert with the larger lambda wins."""
    cfg, om, tables = _om(N=1, E=2, M=2, k=1)
    lam = np.array([[0.2, 0.5]], np.float32)
    rho = np.array([[0.3, 0.7]], np.float32)
    place = np.array([[1, 1]], np.uint16)
    size = np.ones((1, 2))
    cap = np.array([2.0, 1.0])
    new, added = O.replicate(om, lam, rho, size, cap, place)
    assert added == 1 and list(new[0]) == [1, 3]
