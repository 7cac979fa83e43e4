"""Shared builders for oracle tests (host only)."""
from __future__ import annotations

import numpy as np

from oracle import oracle as O
from paper_2608_00573_gb300 import workload as W


def toy_model(spec: dict, H: int | None = None, **table_over) -> O.OracleModel:
    m = spec
    cfg = W.WorkloadConfig(
        name="toy", N=m["N"], d=m["d"], E=m["E"], k=m["k"], F=m["F"], F_sh=m["F_sh"], C=m["C"],
        M=m["M"], H=H if H is not None else m["H"], act=m["act"], renorm_topk=m["renorm_topk"],
        n_sub=m["n_sub"], omega_T=m["omega_T"], omega_D=m["omega_D"], phi_beta=m["phi_beta"])
    N, E, d, C = cfg.N, cfg.E, cfg.d, cfg.C
    tables = dict(
        place=np.array(m["place"], np.uint16), sim=np.array(m["sim"], np.float32),
        sub_thresh=np.array(m["sub_thresh"], np.float32), trans=np.array(m["trans"], np.float32),
        comp=np.array(m["comp"], np.float32), P=np.array(m["P"], np.float32),
        theta=np.array(m["theta"], np.float32), lam=np.array(m["lam"], np.float32),
        eps=np.array(m["eps"], np.float32), d_ref=float(m["d_ref"]))
    tables.update(table_over)
    small = dict(W_r=np.zeros((N, E, d), np.uint16), b_r=np.zeros((N, E), np.float32),
                 W_x=np.zeros((N, C, d), np.uint16), b_x=np.zeros((N, C), np.float32))
    return O.OracleModel(cfg, tables, small)


def small_cfg(**kw) -> W.WorkloadConfig:
    base = dict(name="small", N=4, d=256, E=8, k=2, F=256, F_sh=0, C=1, M=6, H=3,
                act=W.ACT_SWIGLU, renorm_topk=0, T=96, zipf_s=0.5, skip_target=0.2,
                exit_target=0.2, seed=11)
    base.update(kw)
    return W.WorkloadConfig(**base)


def build_small(cfg: W.WorkloadConfig, theta=0.6, exit_bias=1.5, with_experts=True):
    small = W.make_small_weights(cfg, calib={"exit_bias": [exit_bias] * cfg.N})
    tables = W.make_tables(cfg, small["W_r"], calib={"theta": [theta] * cfg.N})
    experts = W.make_expert_weights_host(cfg) if with_experts else None
    return O.OracleModel(cfg, tables, small, experts), tables, small, experts


def bf16_round(x: np.ndarray) -> np.ndarray:
    return W.bf16_bits_to_f32(W.f32_to_bf16_bits(np.asarray(x, dtype=np.float32)))
