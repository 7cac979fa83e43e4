"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test checks the oracle against something other than itself: hand-worked
values (tests/golden), closed forms, brute-force enumeration on tiny inputs,
the paper's guarantees (Properties 2 and 3, constraints (c.5)-(c.10)), and
special cases that reduce to a textbook dense MoE layer.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest

from oracle import oracle as O
from paper_2608_00573_gb300 import workload as W
from tests.oracle_helpers import bf16_round, build_small, small_cfg, toy_model

GOLD = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _toy_spec():
    with open(os.path.join(GOLD, "toy_decisions.json")) as fh:
        return json.load(fh)


# --------------------------------------------------------------------- toy

@pytest.mark.parametrize("case", [c["name"] for c in _toy_spec()["cases"]])
def test_toy_golden(case):
    """Hand-derived decisions for Eq. (30)-(35), (39)-(42) on a 3-server toy."""
    spec = _toy_spec()
    c = next(x for x in spec["cases"] if x["name"] == case)
    over = {}
    if c.get("layer1_place_as_layer0"):
        pl = np.array(spec["model"]["place"], np.uint16)
        pl[1] = pl[0]
        over["place"] = pl
        st = np.array(spec["model"]["sub_thresh"], np.float32)
        st[1] = st[0]
        over["sub_thresh"] = st
    for key, val in c.get("table_over", {}).items():
        over[key] = np.array(val, np.float32)
    if "eps1" in c:
        eps = np.array(spec["model"]["eps"], np.float32)
        eps[1] = c["eps1"]
        over["eps"] = eps
    om = toy_model(spec["model"], H=c["H"], **over)
    ex = c["expect"]
    if "candidates" in ex:
        got = O.candidates(om, c["layer"], c["topk"][0])
        assert [(m, k) for m, k, _ in got] == [(m, k) for m, k, _ in ex["candidates"]]
        np.testing.assert_allclose([q for _, _, q in got], [q for _, _, q in ex["candidates"]], rtol=1e-6)
    if "f" in ex:
        got_f = [O.exec_cost(om, c["layer"], c["s"], m, q, c["Dbar"]) for m, _, q in ex["candidates"]]
        np.testing.assert_allclose(got_f, ex["f"], rtol=1e-6)
    if "phi" in ex:
        tab = O.lookahead_table(om, c["layer"], c["Dbar"] - c["Dhat"], c["Dbar"])
        for key, v in ex["phi"].items():
            m, k = map(int, key.split(","))
            assert tab[m, k] == pytest.approx(v, rel=1e-6)
    D = O.decide_given(om, c["layer"], c["topk"], c["g"], c["I"], c["xi"], c["s"], c["Dhat"],
                       c["Dbar"], c["pJ"], c["last_exec"])
    if "Gamma" in ex:
        assert D.Gamma == pytest.approx(ex["Gamma"], abs=1e-6)
    for key in ("skip_ok", "exit_ok", "action", "s_new"):
        if key in ex:
            assert getattr(D, key) == ex[key], key
    for key in ("tot_exec", "tot_skip", "Dhat_new"):
        if key in ex:
            assert getattr(D, key) == pytest.approx(ex[key], rel=1e-6), key
    if "exp_sel" in ex:
        assert list(D.exp_sel[: len(ex["exp_sel"])]) == ex["exp_sel"]
        assert list(D.srv_sel[: len(ex["srv_sel"])]) == ex["srv_sel"]


# ------------------------------------------------------------------ router

def test_router_matches_sort_and_softmax():
    """Top-k by descending logit (ties to lower index) and I = sum of top-k
    full-softmax gates (Eq. 4), against numpy sort / float64 softmax."""
    cfg = small_cfg(E=16, k=4, d=512)
    om, *_ = build_small(cfg, with_experts=False)
    rng = np.random.default_rng(5)
    h = W.f32_to_bf16_bits(rng.standard_normal((40, cfg.d)).astype(np.float32))
    for l in range(cfg.N):
        Wr = W.bf16_bits_to_f32(om.small["W_r"][l]).astype(np.float64)
        gam = W.bf16_bits_to_f32(om.small["W_norm"][l]).astype(np.float64)
        for t in range(h.shape[0]):
            z, p, topk, g, I = O.router(om, l, h[t])
            hf = W.bf16_bits_to_f32(h[t]).astype(np.float64)
            x = hf / np.sqrt(np.mean(hf * hf) + cfg.norm_eps) * gam       # RMSNorm
            zr = (x @ Wr.T).astype(np.float32) + om.small["b_r"][l]
            np.testing.assert_allclose(z, zr, rtol=0, atol=1e-5)
            order = np.lexsort((np.arange(cfg.E), -z.astype(np.float64)))
            assert list(topk) == list(order[: cfg.k])
            pr = np.exp(z.astype(np.float64) - z.max())
            pr /= pr.sum()
            np.testing.assert_allclose(p, pr, rtol=1e-5, atol=1e-7)
            assert I == pytest.approx(pr[order[: cfg.k]].sum(), rel=1e-5)


def test_importance_is_one_when_k_equals_E():
    """With k = E the activated set is every expert, so I = 1 (Eq. 4)."""
    cfg = small_cfg(E=4, k=4)
    om, *_ = build_small(cfg, with_experts=False)
    rng = np.random.default_rng(1)
    for _ in range(10):
        h = W.f32_to_bf16_bits(rng.standard_normal(cfg.d).astype(np.float32))
        *_, topk, g, I = O.router(om, 0, h)
        assert sorted(topk) == [0, 1, 2, 3]
        assert I == pytest.approx(1.0, abs=2e-7)


def test_router_tie_goes_to_lower_index():
    cfg = small_cfg(E=6, k=2, norm=False)
    om, *_ = build_small(cfg, with_experts=False)
    om.small["W_r"][0][:] = 0          # all logits = bias
    om.small["b_r"][0][:] = np.array([0, 1, 1, 0.5, 1, 0], np.float32)
    h = W.f32_to_bf16_bits(np.ones(cfg.d, np.float32))
    _, _, topk, g, I = O.router(om, 0, h)
    assert list(topk) == [1, 2]


# --------------------------------------------------------------- exit head

def test_exit_head_closed_forms():
    """xi of Eq. (7): sigmoid head (C=1) and max softmax probability (C>1)."""
    d = 64
    for C, b, want in [(1, 0.0, 0.5), (1, math.log(9.0), 0.9), (1, -math.log(3.0), 0.25)]:
        cfg = small_cfg(C=C, d=d)
        om, *_ = build_small(cfg, with_experts=False)
        Wx = np.zeros((C, d), np.uint16)
        xi = O.exit_conf(om, Wx, np.full(C, b, np.float32), W.f32_to_bf16_bits(np.ones(d, np.float32)))
        assert xi == pytest.approx(want, rel=1e-6)
    # C classes with equal logits -> 1/C; one class lifted by delta -> 1/(1+(C-1)e^-delta)
    C = 64
    cfg = small_cfg(C=C, d=d)
    om, *_ = build_small(cfg, with_experts=False)
    Wx = np.zeros((C, d), np.uint16)
    h1 = W.f32_to_bf16_bits(np.ones(d, np.float32))
    assert O.exit_conf(om, Wx, np.zeros(C, np.float32), h1) == pytest.approx(1.0 / C, rel=1e-6)
    b = np.zeros(C, np.float32)
    b[7] = 5.0
    assert O.exit_conf(om, Wx, b, h1) == pytest.approx(1.0 / (1.0 + (C - 1) * math.exp(-5.0)), rel=1e-6)
    # the weights enter through w.h: one-hot h of value 2 and weight 0.5 at that index
    Wx = np.zeros((1, d), np.float32)
    Wx[0, 3] = 0.5
    h = np.zeros(d, np.float32)
    h[3] = 2.0
    cfg = small_cfg(C=1, d=d)
    om, *_ = build_small(cfg, with_experts=False)
    xi = O.exit_conf(om, W.f32_to_bf16_bits(Wx), np.zeros(1, np.float32), W.f32_to_bf16_bits(h), normalise=False)
    assert xi == pytest.approx(1.0 / (1.0 + math.exp(-1.0)), rel=1e-6)
    # RMS-normalised input: mean(h^2) = 4/64, so w.h is scaled by 1/sqrt(1/16 + eps)
    xi = O.exit_conf(om, W.f32_to_bf16_bits(Wx), np.zeros(1, np.float32), W.f32_to_bf16_bits(h), normalise=True)
    x = 1.0 / math.sqrt(1.0 / 16 + cfg.norm_eps)
    assert xi == pytest.approx(1.0 / (1.0 + math.exp(-x)), rel=1e-6)


# -------------------------------------------------------------- candidates

def test_candidate_rules_hold_on_random_tables():
    """Every candidate is deployed (Eq. 11), the exact expert comes first with
    Q = 0 (Eq. 3), substitutes are the n_sub most similar admissible experts."""
    cfg = small_cfg(E=10, M=7, n_sub=3, sub_thresh=-0.2)
    om, tables, *_ = build_small(cfg, with_experts=False)
    place, sim = tables["place"], tables["sim"]
    for l in range(cfg.N):
        for r in range(cfg.E):
            c = O.candidates(om, l, r)
            assert c and c[0][1] == r and c[0][2] == 0.0
            for m, k, q in c:
                assert (place[l, k] >> m) & 1
                if k != r:
                    assert q == pytest.approx(cfg.phi_beta * (1 - sim[l, r, k]) / 2, rel=1e-6)
                    assert q > 0
            exact = [m for m, k, _ in c if k == r]
            assert exact == [m for m in range(cfg.M) if (place[l, r] >> m) & 1]
            subs = sorted({k for _, k, _ in c if k != r})
            elig = [k for k in range(cfg.E) if k != r and sim[l, r, k] >= cfg.sub_thresh]
            assert len(subs) == min(cfg.n_sub, len(elig))
            rest = [k for k in elig if k not in subs]
            if subs and rest:
                assert min(sim[l, r, subs]) >= max(sim[l, r, rest])
            ks = [k for _, k, _ in c if k != r]
            assert ks == sorted(ks)


# -------------------------------------------------------------- look-ahead

@pytest.mark.parametrize("H", [1, 2, 3, 4])
def test_lookahead_table_equals_tree_recursion(H):
    """Memoised Phi^{(H-1)} equals the direct tree recursion of Eq. (39), bit for bit."""
    cfg = small_cfg(E=5, M=4, N=5, H=H)
    om, tables, *_ = build_small(cfg, with_experts=False)
    rng = np.random.default_rng(H)
    for l in range(cfg.N):
        for R, Dbar in [(0.02, 0.02), (0.004, 0.02), (0.0, 0.01), (float(rng.uniform(0, 0.02)), 0.02)]:
            tab = O.lookahead_table(om, l, R, Dbar)
            for m in range(cfg.M):
                for k in range(cfg.E):
                    ref = O.phi_naive(om, l, H - 1, m, k, R, Dbar)
                    assert tab[m, k] == ref, (l, m, k, R)
            if H == 1 or l == cfg.N - 1:
                assert not tab.any()


def test_horizon_one_is_myopic():
    """H = 1: the look-ahead vanishes and the execute choice is argmin f (Sec. V-E)."""
    cfg = small_cfg(E=6, M=5, H=1)
    om, tables, *_ = build_small(cfg, with_experts=False)
    for l in range(cfg.N):
        for r in range(cfg.E):
            for s in range(cfg.M):
                D = O.decide_given(om, l, [r, (r + 1) % cfg.E], [0.6, 0.2], 0.8, -1.0, s, 0.0, 0.02, 0.9, 0)
                cands = O.candidates(om, l, r)
                fs = [O.exec_cost(om, l, s, m, q, 0.02) for m, _, q in cands]
                i = int(np.argmin(fs))
                assert (D.srv_sel[0], D.exp_sel[0]) == (cands[i][0], cands[i][1])


def _bellman_model(seed):
    rng = np.random.default_rng(seed)
    N, E, M = 4, 3, 3
    place = np.zeros((N, E), np.uint16)
    for l in range(N):
        for e in range(E):
            ms = rng.choice(M, size=int(rng.integers(1, 3)), replace=False)
            for m in ms:
                place[l, e] |= 1 << int(m)
    trans = np.zeros((M, M), np.float32)
    for a in range(M):
        for b in range(a + 1, M):
            trans[a, b] = trans[b, a] = np.float32(rng.uniform(1, 30))
    comp = rng.uniform(0.1, 3, size=(N, M)).astype(np.float32)
    sim = rng.uniform(-1, 1, size=(N, E, E)).astype(np.float32)
    route = [int(x) for x in rng.integers(0, E, size=N)]
    P = np.zeros((N - 1, E, E), np.float32)
    for l in range(N - 1):
        P[l, :, route[l + 1]] = 1.0                  # deterministic future routing
    spec = dict(N=N, d=8, E=E, k=1, F=128, F_sh=0, C=1, M=M, H=N, act=1, renorm_topk=0, n_sub=1,
                omega_T=0.5, omega_D=0.5, d_ref=10.0, phi_beta=0.2,
                place=place, sim=sim, sub_thresh=np.full(N, -1.0, np.float32), trans=trans, comp=comp, P=P,
                theta=np.full(N, -1.0, np.float32), lam=np.zeros(N, np.float32),
                eps=np.full(N, 1e30, np.float32))
    return spec, route


@pytest.mark.parametrize("seed", range(8))
def test_bellman_full_horizon_is_optimal(seed):
    """With deterministic transitions, H >= N, no skip/exit and a budget that never
    binds, the look-ahead is exact dynamic programming: the policy's trajectory
    cost equals the brute-force minimum over all (M*|V|)^N trajectories."""
    spec, route = _bellman_model(seed)
    om = toy_model(spec)
    N, M = spec["N"], spec["M"]
    Dbar = 1.0
    s0 = seed % M
    # policy
    s, Dhat, total = s0, 0.0, 0.0
    first_total = None
    for l in range(N):
        D = O.decide_given(om, l, [route[l]], [0.5], 0.5, -1.0, s, Dhat, Dbar, 2.0, 0)
        assert D.action == 0
        total += D.f_sel[0]
        if l == 0:
            first_total = D.tot_exec
        s, Dhat = D.s_new, D.Dhat_new
    # brute force over all trajectories, costs from Eq. (30)-(31) written out
    trans, comp = spec["trans"].astype(np.float64), spec["comp"].astype(np.float64)
    per_layer = []
    for l in range(N):
        r = route[l]
        ks = [r] + [k for k in np.argsort(-spec["sim"][l, r], kind="stable") if k != r][:1]
        opts = []
        for k in ks:
            q = 0.0 if k == r else 0.2 * (1 - float(spec["sim"][l, r, k])) / 2
            for m in range(M):
                if (spec["place"][l, k] >> m) & 1:
                    opts.append((m, k, q))
        per_layer.append(opts)
    best = math.inf
    for traj in itertools.product(*per_layer):
        cur, cost = s0, 0.0
        for l, (m, k, q) in enumerate(traj):
            dly = (trans[cur, m] if m != cur else 0.0) + comp[l, m]
            cost += 0.5 * dly / 10.0 + 0.5 * q / Dbar
            cur = m
        best = min(best, cost)
    assert total == pytest.approx(best, rel=2e-6)
    assert first_total == pytest.approx(best, rel=2e-6)


# ------------------------------------------------- brute-force enumeration

def _py_value(spec, l, h, m, kp, R, Dbar):
    """Future value by explicit enumeration of the action tree (Eq. 39)."""
    N, M = spec["N"], spec["M"]
    best, local = math.inf, False
    cands = spec["cands"][l][kp]
    for (mm, kk, q) in cands:
        if q > R:
            continue
        dly = (spec["trans"][m][mm] if mm != m else 0.0) + spec["comp"][l][mm]
        v = spec["wT"] * dly / spec["d_ref"] + (spec["wD"] * q / Dbar if q > 0 else 0.0)
        if h - 1 > 0 and l < N - 1:
            v += _py_phi(spec, l, h - 1, mm, kk, R, Dbar)
        best = min(best, v)
        local |= mm == m
    if not local and spec["eps"][l] <= R:
        v = spec["wD"] * spec["eps"][l] / Dbar
        if h - 1 > 0 and l < N - 1:
            v += _py_phi(spec, l, h - 1, m, kp, R, Dbar)
        best = min(best, v)
    return best


def _py_phi(spec, l, h, m, k, R, Dbar):
    if h == 0 or l >= spec["N"] - 1:
        return 0.0
    return sum(spec["P"][l][k][kp] * _py_value(spec, l + 1, h, m, kp, R, Dbar) for kp in range(spec["E"]))


@pytest.mark.parametrize("seed,k", [(0, 1), (1, 1), (2, 1), (3, 2), (4, 2), (5, 2)])
def test_decision_matches_bruteforce_enumeration(seed, k):
    """Enumerate every feasible action of Eq. (34) -- all joint execute plans over
    the slots, skip and exit -- with costs (31)/(32) and an explicit look-ahead
    tree, and check the oracle's look-ahead table, totals and choice (Eq. 40).
    k = 1 uses budgets that bind; k = 2 a budget that cannot bind across slots."""
    cfg = small_cfg(E=5, M=4, N=4, k=k, H=3, seed=100 + seed, phi_beta=0.1)
    small = W.make_small_weights(cfg, calib={"exit_bias": [0.0] * cfg.N})
    tables = W.make_tables(cfg, small["W_r"], calib={"theta": [0.5] * cfg.N})
    rng = np.random.default_rng(seed)
    tables["comp"] = rng.uniform(0.5, 8.0, size=tables["comp"].shape).astype(np.float32)
    tables["eps"] = rng.uniform(0.0, 0.06, size=cfg.N).astype(np.float32)
    om = O.OracleModel(cfg, tables, small)
    spec = dict(N=cfg.N, M=cfg.M, E=cfg.E, trans=tables["trans"].astype(np.float64),
                comp=tables["comp"].astype(np.float64), P=tables["P"].astype(np.float64),
                eps=tables["eps"].astype(np.float64), wT=cfg.omega_T, wD=cfg.omega_D, d_ref=tables["d_ref"])
    spec["cands"] = [[O.candidates(om, l, r) for r in range(cfg.E)] for l in range(cfg.N)]
    checked = 0
    for trial in range(40):
        l = int(rng.integers(cfg.N))
        topk = [int(x) for x in rng.choice(cfg.E, size=k, replace=False)]
        g = [0.4, 0.2][:k]
        I = float(np.float32(0.45 if trial % 2 else 0.25))
        s = int(rng.integers(cfg.M))
        if k == 1:
            Dbar = 0.1
            Dhat = float(np.float32(rng.choice([0.0, 0.02, 0.05, 0.08, 0.095])))
        else:
            Dbar, Dhat = 1.0, 0.0
        xi = 0.95 if trial % 3 == 0 else 0.5
        last = 1 if l > 0 else 0
        D = O.decide_given(om, l, topk, g, I, xi, s, Dhat, Dbar, 0.9, last)
        R = float(np.float32(Dbar) - np.float32(Dhat))
        tab = O.lookahead_table(om, l, R, Dbar)
        for m in range(cfg.M):
            for kk in range(cfg.E):
                assert tab[m, kk] == pytest.approx(_py_phi(spec, l, cfg.H - 1, m, kk, R, Dbar), rel=1e-5, abs=1e-6)
        best_plan, best_v = None, math.inf
        plans = [[c for c in spec["cands"][l][r] if Dhat + c[2] <= Dbar] for r in topk]
        for plan in itertools.product(*plans):
            v = 0.0
            for j, (m, kk, q) in enumerate(plan):
                dly = (spec["trans"][s][m] if m != s else 0.0) + spec["comp"][l][m]
                v += cfg.omega_T * dly / spec["d_ref"] + (cfg.omega_D * q / Dbar if q > 0 else 0.0)
                if j == 0:
                    v += _py_phi(spec, l, cfg.H - 1, m, kk, R, Dbar)
            if v < best_v - 1e-9:
                best_v, best_plan = v, plan
        gamma = sum(min((spec["trans"][s][m] if m != s else 0.0) for m, _, _ in p) for p in plans)
        lam = float(tables["lam"][l]) * I
        skip_ok = gamma > 0 and I <= tables["theta"][l] and Dhat + lam <= Dbar
        options = [("exec", best_v)]
        if skip_ok:
            sk = cfg.omega_D * lam / Dbar + _py_phi(spec, l, cfg.H - 1, s, topk[0], R, Dbar)
            options.append(("skip", sk))
            assert D.tot_skip == pytest.approx(sk, rel=1e-5)
        exit_ok = l > 0 and last and xi >= 0.9
        if exit_ok:
            options.append(("exit", 0.0))
        assert bool(D.skip_ok) == bool(skip_ok)
        assert D.tot_exec == pytest.approx(best_v, rel=1e-5)
        vals = sorted(v for _, v in options)
        if len(vals) > 1 and abs(vals[0] - vals[1]) < 1e-5:
            continue                                # a near-tie: order decides
        want = min(options, key=lambda o: o[1])[0]
        got = {0: "exec", 1: "skip", 2: "exit"}[D.action]
        assert got == want
        if want == "exec":
            assert [(D.srv_sel[j], D.exp_sel[j]) for j in range(k)] == [(m, kk) for m, kk, _ in best_plan]
        checked += 1
    assert checked >= 20


# ---------------------------------------------------------- guarantees

def _run_layers(om, tok, h, experts=True):
    rows = []
    for l in range(om.cfg.N):
        h, tok2, out = O.layer_step(om, l, h, tok)
        rows.append((l, tok, tok2, out))
        tok = tok2
    return h, tok, rows


@pytest.mark.parametrize("seed,k,H", [(0, 1, 3), (1, 2, 3), (2, 4, 2), (3, 2, 1)])
def test_paper_guarantees_hold(seed, k, H):
    """Property 2 (budget), Property 3 (exit only at confidence >= p_J after an
    executed layer), and constraints (c.5)-(c.8) on a run with skips and exits."""
    cfg = small_cfg(k=k, H=H, seed=200 + seed, T=128, N=6, E=8, M=10, n_sub=1, sub_thresh=-1.0)
    om, tables, small, ex = build_small(cfg, theta=0.9, exit_bias=1.0)
    tok = W.make_tokens(cfg)
    h = tok.pop("h")
    tok["Dbar"][:] = np.where(np.arange(cfg.T) % 3 == 0, 0.005, 0.02).astype(np.float32)
    seen = np.zeros(4, int)
    prev_action = np.full(cfg.T, -1)
    for l in range(cfg.N):
        before = {kk: v.copy() for kk, v in tok.items()}
        h, tok, out = O.layer_step(om, l, h, tok)
        act = out["action"]
        seen += np.bincount(act, minlength=4)
        # (c.5): dead stays dead; alive only drops by an exit at this layer
        assert np.all(tok["alive"] <= before["alive"])
        assert np.all((act == O.A_DEAD) == (before["alive"] == 0))
        assert np.all((tok["alive"] == 0) == ((before["alive"] == 0) | (act == O.A_EXIT)))
        # Property 2 / (c.10)
        assert np.all(tok["Dhat"] <= tok["Dbar"])
        # Property 3 / (c.9) and (c.6): exit needs an executed previous layer and xi >= p_J
        ex_t = act == O.A_EXIT
        if ex_t.any():
            assert l > 0
            assert np.all(before["last_exec"][ex_t] == 1)
            assert np.all(prev_action[ex_t] == O.A_EXEC)
            assert np.all(out["xi"][ex_t] >= before["pJ"][ex_t])
        # (c.7)/(c.8): one deployed feasible (m, k) per executed slot
        for t in np.nonzero(act == O.A_EXEC)[0]:
            for j in range(k):
                m, e = out["srv_sel"][t * k + j], out["exp_sel"][t * k + j]
                r = out["topk_idx"][t * k + j]
                assert (tables["place"][l, e] >> m) & 1
                assert (m, e) in [(a, b) for a, b, _ in O.candidates(om, l, r)]
        # skip only where execution needs a transmission and I <= theta (Sec. V-C)
        sk = act == O.A_SKIP
        assert np.all(out["Gamma"][sk] > 0)
        assert np.all(out["I"][sk] <= tables["theta"][l])
        assert np.all((out["exp_sel"].reshape(-1, k)[act != O.A_EXEC] == 255))
        prev_action = np.where(act == O.A_DEAD, prev_action, act)
    assert seen[O.A_EXEC] > 0 and seen[O.A_SKIP] > 0 and seen[O.A_EXIT] > 0, seen


def test_full_replication_without_substitutes_runs_local_exact():
    """Every expert on every server and R = {} -> Gamma = 0 always, so no skip,
    and every execution is local and exact (Eq. 30, 35)."""
    cfg = small_cfg(k=2, T=64, placement="full", sub_thresh=float("inf"))
    om, tables, small, ex = build_small(cfg, theta=1.0, exit_bias=-30)
    tok = W.make_tokens(cfg)
    h = tok.pop("h")
    for l in range(cfg.N):
        s_before = tok["s"].copy()
        h, tok, out = O.layer_step(om, l, h, tok)
        assert np.all(out["action"] == O.A_EXEC)
        assert np.all(out["Gamma"] == 0)
        sel = out["exp_sel"].reshape(-1, cfg.k)
        assert np.array_equal(sel, out["topk_idx"].reshape(-1, cfg.k))
        assert np.all(out["srv_sel"].reshape(-1, cfg.k) == s_before[:, None])


def _numpy_dense_moe(cfg, small, ex, h_bits):
    """Textbook top-k MoE forward (router softmax, top-k, expert FFN, weighted sum,
    residual), bf16 storage of act / y / h, float64 arithmetic."""
    h = W.bf16_bits_to_f32(h_bits).astype(np.float64)
    T, d, F, G = h.shape[0], cfg.d, cfg.F, W.GATE_UP_GROUP
    for l in range(cfg.N):
        Wr = W.bf16_bits_to_f32(small["W_r"][l]).astype(np.float64)
        gam = W.bf16_bits_to_f32(small["W_norm"][l]).astype(np.float64)
        xn = h / np.sqrt(np.mean(h * h, axis=1, keepdims=True) + cfg.norm_eps) * gam   # RMSNorm
        z = (xn @ Wr.T).astype(np.float32) + small["b_r"][l]
        xb = bf16_round(xn.astype(np.float32)).astype(np.float64)                   # expert input
        out = h.copy()
        for t in range(T):
            order = np.lexsort((np.arange(cfg.E), -z[t].astype(np.float64)))[: cfg.k]
            p = np.exp(z[t].astype(np.float64) - z[t].max())
            p /= p.sum()
            g = p[order]
            if cfg.renorm_topk:
                g = g / g.sum()
            x = xb[t]
            for j, e in enumerate(order):
                w13 = W.bf16_bits_to_f32(ex["W13"][l, e]).astype(np.float64).reshape(F // G, 2, G, d)
                gate, up = w13[:, 0].reshape(F, d), w13[:, 1].reshape(F, d)
                a = bf16_round(((x @ gate.T) / (1 + np.exp(-(x @ gate.T))) * (x @ up.T)).astype(np.float32))
                y = bf16_round((a.astype(np.float64) @ W.bf16_bits_to_f32(ex["W2"][l, e]).astype(np.float64).T).astype(np.float32))
                out[t] += g[j] * y
            if cfg.F_sh:
                Fs = cfg.F_sh
                w13 = W.bf16_bits_to_f32(ex["W13_sh"][l]).astype(np.float64).reshape(Fs // G, 2, G, d)
                gate, up = w13[:, 0].reshape(Fs, d), w13[:, 1].reshape(Fs, d)
                a = bf16_round(((x @ gate.T) / (1 + np.exp(-(x @ gate.T))) * (x @ up.T)).astype(np.float32))
                out[t] += bf16_round((a.astype(np.float64) @ W.bf16_bits_to_f32(ex["W2_sh"][l]).astype(np.float64).T).astype(np.float32))
        h = bf16_round(out.astype(np.float32)).astype(np.float64)
    return h


@pytest.mark.parametrize("renorm,F_sh", [(1, 0), (0, 128)])
def test_no_skip_no_exit_infinite_budget_equals_dense_moe(renorm, F_sh):
    """No skip, no exit, no substitutes and a budget that cannot bind reduce the
    method to a dense top-k MoE forward (Sec. III-B/C with delta = 0, y = 1)."""
    cfg = small_cfg(N=3, d=256, E=8, k=2, F=256, F_sh=F_sh, renorm_topk=renorm, T=24,
                    sub_thresh=float("inf"), seed=77)
    om, tables, small, ex = build_small(cfg, theta=-1.0, exit_bias=-30)
    tok = W.make_tokens(cfg)
    h0 = tok.pop("h")
    tok["pJ"][:] = 2.0
    tok["Dbar"][:] = np.inf
    h_or, tok_or = O.forward(om, h0, tok)
    assert np.all(tok_or["alive"] == 1) and np.all(tok_or["exit_layer"] == cfg.N)
    ref = _numpy_dense_moe(cfg, small, ex, h0)
    got = W.bf16_bits_to_f32(h_or).astype(np.float64)
    err = np.abs(got - ref).max(axis=1) / np.abs(ref).max(axis=1)
    assert err.max() < 1e-2, err.max()


def test_compaction_is_stable_sort_by_expert():
    cfg = small_cfg(k=2, T=200, N=2)
    om, *_ = build_small(cfg, theta=0.7, exit_bias=1.0)
    tok = W.make_tokens(cfg)
    h = tok.pop("h")
    for l in range(cfg.N):
        h, tok, out = O.layer_step(om, l, h, tok)
        act = out["action"]
        ex_t = np.nonzero(act == O.A_EXEC)[0]
        codes = np.array([t * cfg.k + j for t in ex_t for j in range(cfg.k)], np.int64)
        keys = out["exp_sel"][codes] if codes.size else np.zeros(0, np.int64)
        order = codes[np.argsort(keys, kind="stable")]
        P = codes.size
        assert np.array_equal(out["perm"][:P], order)
        counts = np.bincount(keys, minlength=cfg.E) if P else np.zeros(cfg.E, int)
        assert np.array_equal(out["group_off"][: cfg.E + 1], np.concatenate([[0], np.cumsum(counts)]))


@pytest.mark.parametrize("act,F", [(W.ACT_SWIGLU, 256), (W.ACT_RELU, 256)])
def test_ffn_row_against_float64_matmul(act, F):
    """Expert FFN of one row vs a float64 numpy matmul chain with bf16-rounded
    intermediates (error far below the 2e-2 hidden-state tolerance)."""
    rng = np.random.default_rng(3)
    d = 128
    n13 = 2 if act == W.ACT_SWIGLU else 1
    w13 = W.f32_to_bf16_bits((rng.standard_normal((n13 * F, d)) / math.sqrt(d)).astype(np.float32))
    w2 = W.f32_to_bf16_bits((rng.standard_normal((d, F)) / math.sqrt(F)).astype(np.float32))
    x = W.f32_to_bf16_bits(rng.standard_normal(d).astype(np.float32))
    y = W.bf16_bits_to_f32(O.ffn_row(d, F, act, w13, w2, x)).astype(np.float64)
    xf = W.bf16_bits_to_f32(x).astype(np.float64)
    W13 = W.bf16_bits_to_f32(w13).astype(np.float64)
    if act == W.ACT_SWIGLU:
        G = W.GATE_UP_GROUP
        w = W13.reshape(F // G, 2, G, d)
        gt, up = xf @ w[:, 0].reshape(F, d).T, xf @ w[:, 1].reshape(F, d).T
        a = gt / (1 + np.exp(-gt)) * up
    else:
        a = np.maximum(xf @ W13.T, 0)
    ref = a @ W.bf16_bits_to_f32(w2).astype(np.float64).T
    assert np.abs(y - ref).max() / np.abs(ref).max() < 2e-2 / 4
