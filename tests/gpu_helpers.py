"""Teacher-forced GPU-vs-oracle comparison of one layer (shared by the GPU tests).

Protocol (per layer): the oracle receives the GPU's hidden states and token
state from before the layer, both sides run the layer, and
  * integer outcomes (top-k, action, executed expert and server, next server,
    alive, exit layer, last-executed flag) must be identical except on tokens the
    oracle flags as near a threshold (|score - threshold| <= 1e-5); such tokens
    are counted and must stay under 0.1% of the live tokens;
  * Dhat must be identical after executions and within 1e-6 after a skip;
  * the compaction order and group offsets must be identical when no token
    differs;
  * hidden rows of executed/skipped tokens: max|h_gpu - h_ref| / max|h_ref| <= 2e-2;
    rows of exited or dead tokens (and skipped rows without a shared expert) must
    be bit-identical to the input.
"""
from __future__ import annotations

import numpy as np

from oracle import oracle as O
from paper_2608_00573_gb300 import binding as B
from paper_2608_00573_gb300 import workload as W

HIDDEN_TOL = 2e-2
NEAR_SHARE = 1e-3


def make_engine(cfg, T_max=None, device_experts=False, profile=False, theta=None, exit_bias=None,
                experts=None):
    """Engine + oracle on the seeded workload; theta / exit_bias override the
    calibrated skip thresholds and exit-head biases (every layer)."""
    small = W.make_small_weights(cfg, calib="auto" if exit_bias is None else {"exit_bias": [exit_bias] * cfg.N})
    tables = W.make_tables(cfg, small["W_r"], calib="auto" if theta is None else {"theta": [theta] * cfg.N})
    if experts is None:
        experts = W.make_expert_weights_device(cfg) if device_experts else W.make_expert_weights_host(cfg)
        device_experts = device_experts
    else:
        device_experts = True
    eng = B.Engine(cfg, tables, small, experts, T_max=T_max or cfg.T, profile=profile)
    om = O.OracleModel(cfg, tables, small, None if device_experts else experts)
    return eng, om, tables, small, experts


def experts_layer_host(experts, l):
    """Layer l's expert weights as uint16 numpy (from numpy or device torch tensors)."""
    out = {}
    for k, v in experts.items():
        if v is None:
            continue
        x = v[l]
        if hasattr(x, "detach"):
            import torch
            x = x.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
        out[k] = np.ascontiguousarray(x)
    return out


def compare_layer(cfg, om, eng, l, dev_tok, experts, row_sample=None, check_perm=True):
    import torch
    T = dev_tok["s"].shape[0]
    K, E = cfg.k, cfg.E
    before = B.Engine.tokens_to_host(dev_tok)
    out = eng.alloc_layer_out(T)
    eng.layer_step(l, dev_tok, out=out)
    torch.cuda.synchronize()
    after = B.Engine.tokens_to_host(dev_tok)
    g = {k: (v.view(torch.int16).cpu().numpy().view(np.uint16) if v.dtype == torch.bfloat16 else v.cpu().numpy())
         for k, v in out.items() if v is not None}
    h_in = before.pop("h")
    mask = None
    if row_sample is not None:
        mask = np.zeros(T, np.uint8)
        mask[np.asarray(row_sample)] = 1
    ex_l = experts_layer_host(experts, l)
    hm_gpu = None
    attn_err = 0.0
    if cfg.attn_heads:
        # Attention sublayer: the GPU's h_mid against the oracle's on the live
        # (sampled) rows; the MoE part of the oracle then reads the GPU's h_mid.
        hm_gpu = g["h_attn"]
        amask = (before["alive"] > 0) & (mask.astype(bool) if mask is not None else True)
        hm_or = O.attention(om, l, h_in, before["alive"], experts_l=ex_l, row_mask=amask.astype(np.uint8))
        if amask.any():
            a = W.bf16_bits_to_f32(hm_gpu[amask]).astype(np.float64)
            b = W.bf16_bits_to_f32(hm_or[amask]).astype(np.float64)
            attn_err = float((np.abs(a - b).max(axis=1) / np.maximum(np.abs(b).max(axis=1), 1e-30)).max())
            assert attn_err <= HIDDEN_TOL, f"layer {l}: attention rel err {attn_err}"
    h_or, tok_or, o = O.layer_step(om, l, h_in, before, experts_l=ex_l, row_mask=mask, h_mid=hm_gpu)

    def rows_differ(a, b):
        return (np.asarray(a).reshape(T, -1) != np.asarray(b).reshape(T, -1)).any(axis=1)

    mis = (rows_differ(g["action"], o["action"]) | rows_differ(g["topk_idx"], o["topk_idx"])
           | rows_differ(g["exp_sel"], o["exp_sel"]) | rows_differ(g["srv_sel"], o["srv_sel"])
           | (after["s"] != tok_or["s"]) | (after["alive"] != tok_or["alive"])
           | (after["exit_layer"] != tok_or["exit_layer"]) | (after["last_exec"] != tok_or["last_exec"])
           | (g["lhat"] != o["lhat"]))
    near = o["near"] > 0
    live = before["alive"] > 0
    bad = mis & ~near
    if bad.any():
        t = int(np.nonzero(bad)[0][0])
        raise AssertionError(
            f"layer {l}: {int(bad.sum())} tokens differ away from thresholds; token {t}: "
            f"gpu action {g['action'][t]} topk {g['topk_idx'][t*K:(t+1)*K]} exp {g['exp_sel'][t*K:(t+1)*K]} "
            f"srv {g['srv_sel'][t*K:(t+1)*K]} | oracle action {o['action'][t]} topk {o['topk_idx'][t*K:(t+1)*K]} "
            f"exp {o['exp_sel'][t*K:(t+1)*K]} srv {o['srv_sel'][t*K:(t+1)*K]} I {o['I'][t]} xi {o['xi'][t]} "
            f"gpu I {g['I'][t]} xi {g['xi'][t]} tot_exec {o['tot_exec'][t]} tot_skip {o['tot_skip'][t]}")
    n_live = int(live.sum())
    n_mis = int(mis.sum())
    assert n_mis <= NEAR_SHARE * max(n_live, 1), f"layer {l}: {n_mis} near-threshold mismatches of {n_live}"
    same = ~mis
    act = o["action"]
    # real-valued router / head outputs
    lv = same & live
    assert np.allclose(g["I"][lv], o["I"][lv], rtol=0, atol=2e-6), "importance I"
    xv = lv & (o["xi"] >= 0)
    assert np.allclose(g["xi"][xv], o["xi"][xv], rtol=0, atol=2e-6), "exit confidence"
    assert np.array_equal(g["xi"][lv] >= 0, o["xi"][lv] >= 0)
    # budget state
    ex = same & (act != O.A_SKIP)
    assert np.array_equal(after["Dhat"][ex], tok_or["Dhat"][ex]), "Dhat after execute"
    sk = same & (act == O.A_SKIP)
    if sk.any():
        assert np.abs(after["Dhat"][sk] - tok_or["Dhat"][sk]).max() <= 1e-6, "Dhat after skip"
    assert np.all(after["Dhat"][live] <= after["Dbar"][live]), "Property 2 on the GPU"
    # compaction
    if check_perm and n_mis == 0:
        assert np.array_equal(g["group_off"], o["group_off"]), "group offsets"
        P = int(o["group_off"][E + 1])
        assert np.array_equal(g["perm"][:P], o["perm"][:P]), "compaction order"
    # hidden states
    hg = W.bf16_bits_to_f32(after["h"]).astype(np.float64)
    ho = W.bf16_bits_to_f32(h_or).astype(np.float64)
    hi = W.bf16_bits_to_f32(h_in).astype(np.float64)
    run = same & ((act == O.A_EXEC) | ((act == O.A_SKIP) & (cfg.F_sh > 0)))
    if mask is not None:
        run &= mask.astype(bool)
    err = 0.0
    if run.any():
        num = np.abs(hg[run] - ho[run]).max(axis=1)
        den = np.maximum(np.abs(ho[run]).max(axis=1), 1e-30)
        err = float((num / den).max())
        assert err <= HIDDEN_TOL, f"layer {l}: hidden rel err {err}"
    still = same & ((act == O.A_EXIT) | (act == O.A_DEAD))
    assert np.array_equal(after["h"][still], h_in[still]), "untouched rows changed"
    bare_skip = same & (act == O.A_SKIP) & (cfg.F_sh == 0)
    assert np.array_equal(after["h"][bare_skip], (hm_gpu if hm_gpu is not None else h_in)[bare_skip]), \
        "skipped rows must carry the MoE input unchanged"
    counts = np.bincount(g["action"], minlength=4)
    return dict(layer=l, live=n_live, near_mismatch=n_mis, near=int(near.sum()), max_rel_err=err,
                attn_rel_err=attn_err,
                exec=int(counts[0]), skip=int(counts[1]), exit=int(counts[2]), dead=int(counts[3]),
                rows_checked=int(run.sum()), oracle_out=o, s_before=before["s"])
