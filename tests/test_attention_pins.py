"""Pins of the oracle's attention sublayer (the full block: Sec. III-C, attention
placement, with the pre-norm grouped-query attention of the model families of
Sec. VI-A).

The oracle is checked against closed forms (first position of a sequence,
zero keys), the rotary embedding's defining properties, causality and
sequence isolation, torch's scaled-dot-product attention on a tiny case, and
the special case of a zero output projection, where the full block must equal
the MoE step alone.
"""
import math

import numpy as np
import pytest

from oracle import oracle as O
from paper_2608_00573_gb300 import workload as W
from tests.oracle_helpers import build_small, small_cfg


def _cfg(**kw):
    base = dict(name="attn", N=2, d=64, E=4, k=2, F=64, T=24, M=4, attn_heads=4, attn_kv_heads=2,
                head_dim=16, attn_seq=8, rope_theta=10000.0, seed=31)
    base.update(kw)
    return small_cfg(**base)


def _bf(x):
    """float64 -> float32 -> bf16, the rounding the oracle applies."""
    return W.bf16_bits_to_f32(W.f32_to_bf16_bits(np.asarray(x, dtype=np.float64).astype(np.float32))).astype(
        np.float64)


def _f(bits):
    return W.bf16_bits_to_f32(bits).astype(np.float64)


def _attn_input(cfg, small, h, l):
    hf = _f(h)
    r = 1.0 / np.sqrt((hf * hf).mean(axis=1, keepdims=True) + cfg.norm_eps)
    return _bf(hf * r * _f(small["W_attn_norm"][l]))


def _close_bf16(got_bits, want, min_exact=0.99):
    """Equal up to the rounding order of the double sums: nearly every element is
    bit-identical and none is off by more than one bf16 step."""
    g = _f(got_bits)
    w = np.asarray(want, dtype=np.float64)
    exact = (g == w).mean()
    step = np.maximum(np.abs(w), 1e-30) * 2.0 ** -7
    assert exact >= min_exact, exact
    assert np.all(np.abs(g - w) <= step + 1e-30)


def test_rope_properties():
    rng = np.random.default_rng(0)
    Dh, theta = 16, 10000.0
    q, k = rng.standard_normal(Dh), rng.standard_normal(Dh)
    assert np.array_equal(O.rope(q, 0, theta), q)
    for p in (1, 5, 127):
        assert np.linalg.norm(O.rope(q, p, theta)) == pytest.approx(np.linalg.norm(q), rel=1e-12)
    # scores depend on the relative position only
    for p, pp, sh in [(3, 1, 7), (10, 10, 2), (0, 9, 100)]:
        a = O.rope(q, p, theta) @ O.rope(k, pp, theta)
        b = O.rope(q, p + sh, theta) @ O.rope(k, pp + sh, theta)
        assert a == pytest.approx(b, rel=1e-10, abs=1e-12)
    # unit vector of pair i turns by pos * theta^(-2i/Dh) into the (i, i + Dh/2) plane
    for i in (0, 3, 7):
        e = np.zeros(Dh)
        e[i] = 1.0
        y = O.rope(e, 6, theta)
        ang = 6 * theta ** (-2.0 * i / Dh)
        want = np.zeros(Dh)
        want[i], want[i + Dh // 2] = math.cos(ang), math.sin(ang)
        assert np.allclose(y, want, atol=1e-15)


def test_first_position_attends_to_itself_only():
    """At position 0 the softmax has one key: o = v of the token's key/value
    head, so h_mid = bf16(h + o W_o^T) in closed form."""
    cfg = _cfg()
    om, tables, small, experts = build_small(cfg)
    tok = W.make_tokens(cfg)
    h = tok["h"]
    hm = O.attention(om, 0, h, tok["alive"])
    a = _attn_input(cfg, small, h, 0)
    Wqkv = _f(experts["W_qkv"][0])
    Wo = _f(experts["W_o"][0])
    nq, nkv, Dh = cfg.attn_heads * cfg.head_dim, cfg.attn_kv_heads * cfg.head_dim, cfg.head_dim
    grp = cfg.attn_heads // cfg.attn_kv_heads
    for t in range(0, cfg.T, cfg.attn_seq):
        v = _bf(a[t] @ Wqkv[nq + nkv:].T)
        o = np.concatenate([v[(hq // grp) * Dh:(hq // grp + 1) * Dh] for hq in range(cfg.attn_heads)])
        _close_bf16(hm[t], _bf(_f(h[t]) + o @ Wo.T), min_exact=0.95)


def test_zero_keys_average_the_values():
    """With the key projection zero every score is 0, so each token averages
    the values of its sequence up to itself (uniform causal weights)."""
    cfg = _cfg()
    om, tables, small, experts = build_small(cfg)
    nq, nkv = cfg.attn_heads * cfg.head_dim, cfg.attn_kv_heads * cfg.head_dim
    ex = {k: v.copy() for k, v in experts.items()}
    ex["W_qkv"][0][nq:nq + nkv] = 0
    om = O.OracleModel(cfg, tables, small, ex)
    tok = W.make_tokens(cfg)
    h = tok["h"]
    hm = O.attention(om, 0, h, tok["alive"])
    a = _attn_input(cfg, small, h, 0)
    V = _bf(a @ _f(ex["W_qkv"][0])[nq + nkv:].T)
    Wo = _f(ex["W_o"][0])
    Dh, grp = cfg.head_dim, cfg.attn_heads // cfg.attn_kv_heads
    want = np.zeros((cfg.T, cfg.d))
    for t in range(cfg.T):
        j0 = t - t % cfg.attn_seq
        mean = V[j0:t + 1].mean(axis=0)
        o = _bf(np.concatenate([mean[(hq // grp) * Dh:(hq // grp + 1) * Dh] for hq in range(cfg.attn_heads)]))
        want[t] = _bf(_f(h[t]) + o @ Wo.T)
    _close_bf16(hm, want, min_exact=0.95)


def test_causal_and_isolated_sequences():
    """Changing token 3 of the first sequence changes only that sequence's
    tokens from position 3 on."""
    cfg = _cfg()
    om, *_ = build_small(cfg)
    tok = W.make_tokens(cfg)
    h = tok["h"]
    base = O.attention(om, 0, h, tok["alive"])
    h2 = h.copy()
    h2[3] = W.f32_to_bf16_bits(np.random.default_rng(1).standard_normal(cfg.d).astype(np.float32))
    got = O.attention(om, 0, h2, tok["alive"])
    S = cfg.attn_seq
    assert np.array_equal(got[:3], base[:3])
    assert np.array_equal(got[S:], base[S:])
    assert all((got[t] != base[t]).any() for t in range(4, S))


def test_keys_of_tokens_that_left_still_count():
    """A token that is no longer live keeps its row (h_mid = h) but its key and
    value still feed the later tokens of its sequence."""
    cfg = _cfg()
    om, *_ = build_small(cfg)
    tok = W.make_tokens(cfg)
    h = tok["h"]
    alive = tok["alive"].copy()
    alive[2] = 0
    got = O.attention(om, 0, h, alive)
    ref = O.attention(om, 0, h, tok["alive"])
    assert np.array_equal(got[2], h[2])
    mask = np.ones(cfg.T, bool)
    mask[2] = False
    assert np.array_equal(got[mask], ref[mask])


def test_matches_torch_scaled_dot_product_attention():
    """The whole sublayer against torch: projections with matmul, the rotary
    embedding as a complex rotation of the projected query and key heads
    (rounded to bf16 once, after the rotation), causal attention by
    scaled_dot_product_attention with the key/value heads repeated."""
    torch = pytest.importorskip("torch")
    cfg = _cfg(T=20)                     # a full sequence of 8 and a ragged 4
    om, tables, small, experts = build_small(cfg)
    tok = W.make_tokens(cfg)
    h = tok["h"]
    hm = O.attention(om, 0, h, tok["alive"])
    a = torch.tensor(_attn_input(cfg, small, h, 0))
    Hq, Hkv, Dh, S = cfg.attn_heads, cfg.attn_kv_heads, cfg.head_dim, cfg.attn_seq
    Wqkv = torch.tensor(_f(experts["W_qkv"][0]))
    Wo = torch.tensor(_f(experts["W_o"][0]))

    def rnd(x):
        return torch.tensor(_bf(x.numpy()))

    qkv = a @ Wqkv.T
    q = qkv[:, :Hq * Dh].reshape(-1, Hq, Dh)
    k = qkv[:, Hq * Dh:(Hq + Hkv) * Dh].reshape(-1, Hkv, Dh)
    v = rnd(qkv[:, (Hq + Hkv) * Dh:].reshape(-1, Hkv, Dh))
    pos = torch.arange(cfg.T, dtype=torch.float64) % S
    inv = cfg.rope_theta ** (-2.0 * torch.arange(Dh // 2, dtype=torch.float64) / Dh)
    rot = torch.polar(torch.ones(cfg.T, Dh // 2, dtype=torch.float64), pos[:, None] * inv[None, :])

    def rope(x):
        z = torch.complex(x[..., :Dh // 2], x[..., Dh // 2:]) * rot[:, None, :]
        return rnd(torch.cat([z.real, z.imag], dim=-1))

    q, k = rope(q), rope(k)
    out = torch.zeros(cfg.T, Hq * Dh, dtype=torch.float64)
    for s0 in range(0, cfg.T, S):
        s1 = min(s0 + S, cfg.T)
        qs = q[s0:s1].transpose(0, 1)
        ks = k[s0:s1].transpose(0, 1).repeat_interleave(Hq // Hkv, dim=0)
        vs = v[s0:s1].transpose(0, 1).repeat_interleave(Hq // Hkv, dim=0)
        o = torch.nn.functional.scaled_dot_product_attention(qs, ks, vs, is_causal=True)
        out[s0:s1] = o.transpose(0, 1).reshape(s1 - s0, Hq * Dh)
    want = _bf((torch.tensor(_f(h)) + rnd(out) @ Wo.T).numpy())
    _close_bf16(hm, want, min_exact=0.95)


def test_zero_output_projection_reduces_to_the_moe_step():
    """With W_o = 0 the attention adds nothing (h_mid = h): the full block's
    decisions and outputs equal those of the MoE step alone."""
    cfg = _cfg(d=256, E=8, F=256, T=64, attn_heads=4, attn_kv_heads=4, head_dim=64, attn_seq=16, N=3)
    om, tables, small, experts = build_small(cfg, theta=0.9, exit_bias=1.0)
    ex = {k: v.copy() for k, v in experts.items()}
    ex["W_o"][:] = 0
    om_blk = O.OracleModel(cfg, tables, small, ex)
    om_moe = O.OracleModel(cfg.replace(attn_heads=0), tables, small, ex)
    tok = W.make_tokens(cfg)
    h0 = tok.pop("h")
    ha, ta = h0, dict(tok)
    hb, tb = h0, dict(tok)
    for l in range(cfg.N):
        ha, ta, oa = O.layer_step(om_blk, l, ha, ta)
        hb, tb, ob = O.layer_step(om_moe, l, hb, tb)
        for key in ("action", "exp_sel", "srv_sel", "topk_idx", "perm", "group_off"):
            assert np.array_equal(oa[key], ob[key]), key
        assert np.array_equal(ha, hb)
        assert np.array_equal(ta["Dhat"], tb["Dhat"])


def test_full_block_exit_keeps_the_entering_state():
    """A token that exits at layer l leaves with the state that entered the
    layer; an executed or skipped one with the post-attention state plus its
    FFN output (a skip without a shared expert: the post-attention state)."""
    cfg = _cfg(d=256, E=8, F=256, T=64, M=10, n_sub=1, attn_heads=4, attn_kv_heads=2, head_dim=64,
               attn_seq=16, N=4)
    om, tables, small, experts = build_small(cfg, theta=0.9, exit_bias=1.0)
    tok = W.make_tokens(cfg)
    h = tok.pop("h")
    seen = {O.A_EXIT: 0, O.A_SKIP: 0}
    n_xi = 0
    for l in range(cfg.N):
        hm = O.attention(om, l, h, tok["alive"])
        h_out, tok2, out = O.layer_step(om, l, h, tok)
        # the exit head of layer l-1 reads the state entering layer l (sigmoid
        # head on the RMS-normalised state, Eq. 7), not the post-attention one
        if l > 0:
            w = _f(small["W_x"][l - 1][0])
            for t in np.nonzero(out["xi"] >= 0)[0]:
                hf = _f(h[t])
                x = np.float32(hf @ w / np.sqrt((hf * hf).mean() + cfg.norm_eps)) + small["b_x"][l - 1][0]
                want = np.float32(1.0) / (np.float32(1.0) + np.exp(-np.float32(x)))
                assert out["xi"][t] == pytest.approx(want, abs=1e-6)
                n_xi += 1
        h_out2, _, _ = O.layer_step(om, l, h, tok, h_mid=hm)
        assert np.array_equal(h_out, h_out2)
        for t in range(cfg.T):
            a = out["action"][t]
            if a == O.A_EXIT:
                assert np.array_equal(h_out[t], h[t])
                seen[a] += 1
            elif a == O.A_SKIP:
                assert np.array_equal(h_out[t], hm[t])
                seen[a] += 1
            elif a == O.A_DEAD:
                assert np.array_equal(h_out[t], h[t])
        h, tok = h_out, tok2
    assert seen[O.A_EXIT] > 0 and seen[O.A_SKIP] > 0 and n_xi > 0, (seen, n_xi)
