"""Seeded synthetic workloads for the adaptive-depth MoE step.

This module only draws inputs: weights, placement, cost tables, transition
statistics, thresholds and the initial per-token state.  It holds none of the
method's arithmetic (no router, no softmax, no cost, no look-ahead, no FFN), so
both the CUDA library and the CPU oracle can consume the same draws.

Shapes stand in for the three models the paper evaluates (Sec. VI-A:
Switch-Base-8E, Qwen-MoE-A2.7B, Mixtral-8x7B); the paper's weights, datasets
and testbed are not available, so every value here is synthetic:

* weights ~ N(0, 1/fan_in) stored as bf16 (attention projections included);
  hidden states ~ N(0, 1) in bf16;
  RMSNorm weights of the MoE sublayer ~ N(1, 0.1^2) in bf16 (all three models
  are pre-norm; without the norm a random-weight SwiGLU stack overflows bf16
  within about ten layers), and likewise for the attention sublayer;
* router bias b_e = -s * ln(e + 1), which makes expert popularity Zipf(s);
* users are blocks of 128 tokens; each user's access server a(i) (Eq. 12) is
  drawn Zipf(1.0) over the M servers, with p_J = 0.9 and a per-token budget
  Dbar = budget (Eq. 33, default 2% as in Sec. VI-A);
* the cost matrix is symmetric with a zero diagonal: U[1, 50] ms for the tiny
  case, otherwise z/B + tau with z = 2d bytes, B ~ U[0.8, 10] Gbps and
  tau ~ U[0.3, 22] ms (the link ranges of Sec. VI-A);
* compute delay comp[l][m] = c_l / F_m (Eq. 15) with c_l the FLOPs of one
  expert on one token and F_m ~ U[18, 120] TFLOPS (Sec. VI-A);
* transition rows P_l(k -> .) ~ Dirichlet(1) (Eq. 38);
* expert similarity Sim_l = cosine similarity of the router rows of layer l;
* skip thresholds theta_l and exit-head biases come from a calibration file
  written by a script that runs only the oracle (see ``workload_calib.json``);
  without an entry they default to "no skips, no exits".

Large expert weights are drawn on the device with torch's seeded generator;
small configurations are drawn on the host with numpy.
"""
from __future__ import annotations

import dataclasses
import json
import math
import os
from typing import Optional

import numpy as np

CALIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "workload_calib.json")

# Row interleave of the gate/up projection in W13: rows [256b, 256b+128) hold
# gate rows 128b..128b+127 and rows [256b+128, 256b+256) the matching up rows.
GATE_UP_GROUP = 128

ACT_RELU = 0
ACT_SWIGLU = 1


@dataclasses.dataclass
class WorkloadConfig:
    name: str
    N: int            # MoE layers
    d: int            # d_model
    E: int            # routed experts per layer
    k: int            # top-k
    F: int            # routed expert d_ff
    F_sh: int = 0     # shared expert d_ff (0 = none)
    C: int = 1        # exit-head classes (1 = sigmoid head)
    M: int = 10       # simulated servers
    H: int = 3        # look-ahead horizon
    act: int = ACT_SWIGLU
    renorm_topk: int = 0
    T: int = 64
    zipf_s: float = 0.0
    budget: float = 0.02
    p_J: float = 0.9
    placement: str = "replicas"      # "replicas" (2-4 per expert) | "subset3"
    trans: str = "link"              # "link" | "uniform"
    n_sub: int = 3
    phi_beta: float = 0.02
    sub_thresh: float = -1.0
    omega_T: float = 0.5
    omega_D: float = 0.5
    skip_target: float = 0.0         # target fraction of layer-tokens skipped
    exit_target: float = 0.0         # target fraction of tokens exited
    exit_peak: Optional[float] = None
    exit_width: float = 2.0
    norm: bool = True                # pre-FFN RMSNorm of the MoE sublayer
    norm_eps: float = 1e-6
    n_centroids: int = 0             # K_c centroids per layer for exit prediction (Eq. 36); 0 = off
    # Attention sublayer of the full block (0 heads = the MoE step alone).
    attn_heads: int = 0              # query heads
    attn_kv_heads: int = 0           # key/value heads (grouped-query attention)
    head_dim: int = 0
    attn_seq: int = 128              # tokens per sequence (one user's block)
    rope_theta: float = 1.0e6
    seed: int = 0

    @property
    def n_qkv(self) -> int:
        return (self.attn_heads + 2 * self.attn_kv_heads) * self.head_dim

    @property
    def n13(self) -> int:
        return 2 if self.act == ACT_SWIGLU else 1

    @property
    def n_mat(self) -> int:
        return 3 if self.act == ACT_SWIGLU else 2

    def replace(self, **kw) -> "WorkloadConfig":
        return dataclasses.replace(self, **kw)


# Slope of phi in Q = phi((1 - Sim)/2) (Eq. 3).  The paper takes phi from its
# reference [37], which is not available; 0.001 makes a substitution cost about
# 2.5% of the 2% per-token budget, which reproduces the execution mix the paper
# reports for Mixtral (Fig. 5(b): most executions local, about one in ten
# layer-tokens skipped).
PHI_BETA = 0.001

# The five workloads: four model-shaped forwards and the decode stress case.
CONFIGS = {
    "switch_tiny": WorkloadConfig(
        name="switch_tiny", N=4, d=768, E=8, k=1, F=3072, C=64, act=ACT_RELU, T=64,
        placement="subset3", trans="uniform", skip_target=0.2, exit_target=0.15,
        phi_beta=PHI_BETA, seed=0),
    "switch": WorkloadConfig(
        name="switch", N=12, d=768, E=8, k=1, F=3072, C=64, act=ACT_RELU, T=4096,
        zipf_s=1.2, skip_target=0.20, exit_target=0.15, phi_beta=PHI_BETA, seed=1),
    "qwen": WorkloadConfig(
        name="qwen", N=24, d=2048, E=60, k=4, F=1408, F_sh=5632, C=1, act=ACT_SWIGLU,
        T=8192, zipf_s=1.0, skip_target=0.11, exit_target=0.12, phi_beta=PHI_BETA, seed=2),
    "mixtral": WorkloadConfig(
        name="mixtral", N=32, d=4096, E=8, k=2, F=14336, C=1, act=ACT_SWIGLU, renorm_topk=1,
        T=16384, zipf_s=1.0, skip_target=0.11, exit_target=0.12, exit_peak=21.0,
        phi_beta=PHI_BETA, seed=3),
    "mixtral_decode": WorkloadConfig(
        name="mixtral_decode", N=32, d=4096, E=8, k=2, F=14336, C=1, act=ACT_SWIGLU,
        renorm_topk=1, T=256, zipf_s=1.5, skip_target=0.11, exit_target=0.40,
        exit_peak=18.0, exit_width=4.0, phi_beta=PHI_BETA, seed=4),
}


# Attention shapes of the three model families (query heads, key/value heads,
# head dimension): Switch-Base 12 x 64, Qwen-MoE-A2.7B 16 x 128, Mixtral-8x7B
# 32 query / 8 key-value heads of 128.
ATTN_SHAPES = {"switch": (12, 12, 64), "qwen": (16, 16, 128), "mixtral": (32, 8, 128)}


def with_attention(cfg: WorkloadConfig) -> WorkloadConfig:
    """The workload with the attention sublayer of its model family in front of
    every MoE step (the full transformer block)."""
    fam = next(k for k in ATTN_SHAPES if cfg.name.startswith(k))
    hq, hkv, dh = ATTN_SHAPES[fam]
    return cfg.replace(attn_heads=hq, attn_kv_heads=hkv, head_dim=dh)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bf16 (round to nearest even) and return the raw bits."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    r = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)
    nan = np.isnan(x)
    if nan.any():
        r[nan] = 0x7FC0
    return r


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def _normal_bf16(rng: np.random.Generator, shape, std: float) -> np.ndarray:
    return f32_to_bf16_bits((rng.standard_normal(shape, dtype=np.float32) * np.float32(std)))


def load_calibration(name: str) -> Optional[dict]:
    if not os.path.exists(CALIB_PATH):
        return None
    with open(CALIB_PATH) as fh:
        return json.load(fh).get(name)


def make_tables(cfg: WorkloadConfig, W_r_bits: Optional[np.ndarray] = None,
                calib: Optional[dict] = "auto") -> dict:
    """Placement, similarity, cost, transition and threshold tables (host, numpy)."""
    rng = np.random.default_rng([cfg.seed, 101])
    N, E, M = cfg.N, cfg.E, cfg.M
    # Placement x_{m,l,k} (Eq. 1-2) as a server bit mask per (layer, expert).
    place = np.zeros((N, E), dtype=np.uint16)
    if cfg.placement == "subset3":
        for l in range(N):
            for m in range(M):
                for e in rng.choice(E, size=min(3, E), replace=False):
                    place[l, e] |= np.uint16(1 << m)
            for e in range(E):       # coverage patch (Eq. 2)
                if place[l, e] == 0:
                    place[l, e] = np.uint16(1 << int(rng.integers(M)))
    elif cfg.placement == "full":
        place[:] = np.uint16((1 << M) - 1)
    else:
        for l in range(N):
            for e in range(E):
                r = int(rng.integers(2, 5))
                for m in rng.choice(M, size=min(r, M), replace=False):
                    place[l, e] |= np.uint16(1 << int(m))
    # Server-to-server delay in ms, symmetric with a zero diagonal.
    trans = np.zeros((M, M), dtype=np.float32)
    for a in range(M):
        for b in range(a + 1, M):
            if cfg.trans == "uniform":
                v = rng.uniform(1.0, 50.0)
            else:
                bw = rng.uniform(0.8, 10.0) * 1e9           # bit/s
                tau = rng.uniform(0.3, 22.0)                 # ms
                v = (2 * cfg.d * 8) / bw * 1e3 + tau
            trans[a, b] = trans[b, a] = np.float32(v)
    flops = 2.0 * cfg.n_mat * cfg.d * cfg.F                   # c_l of one expert, one token
    F_m = rng.uniform(18.0, 120.0, size=M) * 1e12
    comp = np.tile((flops / F_m * 1e3).astype(np.float32), (N, 1))
    # Transition statistics P_l(k -> k'), rows ~ Dirichlet(1).
    P = rng.dirichlet(np.ones(E), size=(max(N - 1, 0), E)).astype(np.float32)
    # Router-induced similarity: cosine of router rows.
    if W_r_bits is not None:
        W = bf16_bits_to_f32(W_r_bits).astype(np.float64)
        nrm = np.linalg.norm(W, axis=2, keepdims=True)
        Wn = W / np.maximum(nrm, 1e-30)
        sim = np.einsum("led,lfd->lef", Wn, Wn).astype(np.float32)
    else:
        sim = rng.uniform(-1, 1, size=(N, E, E)).astype(np.float32)
        sim = ((sim + sim.transpose(0, 2, 1)) / 2).astype(np.float32)
        for l in range(N):
            np.fill_diagonal(sim[l], 1.0)
    sub_thresh = np.full(N, cfg.sub_thresh, dtype=np.float32)
    if calib == "auto":
        calib = load_calibration(cfg.name)
    if calib is not None and len(calib.get("theta", [])) == N:
        theta = np.asarray(calib["theta"], dtype=np.float32)
    else:
        theta = np.full(N, -1.0, dtype=np.float32)            # no skips
    # Skip tolerance eps_l = Dbar / kappa (Eq. 25) and linear Lambda = lambda_l * I
    # with lambda_l = eps_l / theta_l so that (24) holds with equality.
    kappa = max(cfg.skip_target * N, 1.0)
    eps = np.full(N, cfg.budget / kappa, dtype=np.float32)
    lam = np.where(theta > 0, eps / np.maximum(theta, 1e-6), eps).astype(np.float32)
    # Reference per-step delay: mean over (source server, expert) of the cheapest
    # exact execution (Eq. 30 with Q = 0), layer 0.
    best = []
    for s in range(M):
        for e in range(E):
            ms = [m for m in range(M) if place[0, e] >> m & 1]
            best.append(min((trans[s, m] if m != s else 0.0) + comp[0, m] for m in ms))
    d_ref = np.float32(np.mean(best))
    return dict(place=place, trans=trans, comp=comp, P=P, sim=sim, sub_thresh=sub_thresh,
                theta=theta, lam=lam, eps=eps, d_ref=float(d_ref))


def make_small_weights(cfg: WorkloadConfig, calib: Optional[dict] = "auto") -> dict:
    """Router, exit-head and norm weights (always host) -- small for every configuration."""
    rng = np.random.default_rng([cfg.seed, 202])
    N, E, d, C = cfg.N, cfg.E, cfg.d, cfg.C
    W_r = _normal_bf16(rng, (N, E, d), 1.0 / math.sqrt(d))
    W_norm = None
    if cfg.norm:
        W_norm = f32_to_bf16_bits((1.0 + 0.1 * np.random.default_rng([cfg.seed, 505]).standard_normal(
            (N, d))).astype(np.float32))
    b_r = np.tile((-cfg.zipf_s * np.log(np.arange(E) + 1.0)).astype(np.float32), (N, 1))
    W_x = _normal_bf16(rng, (N, C, d), 1.0 / math.sqrt(d))
    b_x = np.zeros((N, C), dtype=np.float32)
    if calib == "auto":
        calib = load_calibration(cfg.name)
    if calib is not None and len(calib.get("exit_bias", [])) == N:
        b_x[:, 0] = np.asarray(calib["exit_bias"], dtype=np.float32)
    else:
        b_x[:, 0] = -30.0                                     # no exits
    out = dict(W_r=W_r, b_r=b_r, W_x=W_x, b_x=b_x, W_norm=W_norm)
    if cfg.attn_heads:
        out["W_attn_norm"] = f32_to_bf16_bits((1.0 + 0.1 * np.random.default_rng([cfg.seed, 707]).standard_normal(
            (N, d))).astype(np.float32))
    if cfg.n_centroids:
        out.update(make_centroids(cfg))
    return out


def make_centroids(cfg: WorkloadConfig) -> dict:
    """Synthetic stand-in for the token-similarity reference set (Eq. 36): per
    layer, K_c centroid directions ~ N(0, 1) in bf16 and, per centroid, an
    average exit layer drawn around the workload's exit peak (uniform over the
    remaining depth when it has none), never before the next layer."""
    rng = np.random.default_rng([cfg.seed, 606])
    N, K, d = cfg.N, cfg.n_centroids, cfg.d
    cent = _normal_bf16(rng, (N, K, d), 1.0)
    peak = cfg.exit_peak if cfg.exit_peak is not None else 0.75 * N
    ex = np.zeros((N, K), np.float32)
    for l in range(N):
        v = rng.normal(peak, max(cfg.exit_width, 1.0) * 2.0, size=K)
        ex[l] = np.clip(v, l + 1, N).astype(np.float32)
    return dict(centroids=cent, centroid_exit=ex)


def make_expert_weights_host(cfg: WorkloadConfig) -> dict:
    """Expert weights as bf16 bits on the host (small configurations only)."""
    rng = np.random.default_rng([cfg.seed, 303])
    N, E, d, F = cfg.N, cfg.E, cfg.d, cfg.F
    out = dict(
        W13=_normal_bf16(rng, (N, E, cfg.n13 * F, d), 1.0 / math.sqrt(d)),
        W2=_normal_bf16(rng, (N, E, d, F), 1.0 / math.sqrt(F)),
    )
    if cfg.F_sh:
        out["W13_sh"] = _normal_bf16(rng, (N, 2 * cfg.F_sh, d), 1.0 / math.sqrt(d))
        out["W2_sh"] = _normal_bf16(rng, (N, d, cfg.F_sh), 1.0 / math.sqrt(cfg.F_sh))
    if cfg.attn_heads:
        ra = np.random.default_rng([cfg.seed, 808])
        hd = cfg.attn_heads * cfg.head_dim
        out["W_qkv"] = _normal_bf16(ra, (N, cfg.n_qkv, d), 1.0 / math.sqrt(d))
        out["W_o"] = _normal_bf16(ra, (N, d, hd), 1.0 / math.sqrt(hd))
    return out


def make_expert_weights_device(cfg: WorkloadConfig, device="cuda") -> dict:
    """Expert weights as torch bf16 tensors drawn on the device (torch Philox)."""
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(cfg.seed * 7919 + 303)
    N, E, d, F = cfg.N, cfg.E, cfg.d, cfg.F
    W13 = torch.empty((N, E, cfg.n13 * F, d), dtype=torch.bfloat16, device=device)
    W2 = torch.empty((N, E, d, F), dtype=torch.bfloat16, device=device)
    for l in range(N):
        W13[l].normal_(0.0, 1.0 / math.sqrt(d), generator=g)
        W2[l].normal_(0.0, 1.0 / math.sqrt(F), generator=g)
    out = dict(W13=W13, W2=W2)
    if cfg.F_sh:
        W13_sh = torch.empty((N, 2 * cfg.F_sh, d), dtype=torch.bfloat16, device=device)
        W2_sh = torch.empty((N, d, cfg.F_sh), dtype=torch.bfloat16, device=device)
        for l in range(N):
            W13_sh[l].normal_(0.0, 1.0 / math.sqrt(d), generator=g)
            W2_sh[l].normal_(0.0, 1.0 / math.sqrt(cfg.F_sh), generator=g)
        out.update(W13_sh=W13_sh, W2_sh=W2_sh)
    if cfg.attn_heads:
        ga = torch.Generator(device=device)
        ga.manual_seed(cfg.seed * 7919 + 808)
        hd = cfg.attn_heads * cfg.head_dim
        W_qkv = torch.empty((N, cfg.n_qkv, d), dtype=torch.bfloat16, device=device)
        W_o = torch.empty((N, d, hd), dtype=torch.bfloat16, device=device)
        for l in range(N):
            W_qkv[l].normal_(0.0, 1.0 / math.sqrt(d), generator=ga)
            W_o[l].normal_(0.0, 1.0 / math.sqrt(hd), generator=ga)
        out.update(W_qkv=W_qkv, W_o=W_o)
    return out


def make_tokens(cfg: WorkloadConfig, T: Optional[int] = None, seed_offset: int = 0) -> dict:
    """Initial hidden states and per-token state (Alg. 2 initialisation)."""
    T = cfg.T if T is None else T
    rng = np.random.default_rng([cfg.seed, 404, seed_offset])
    h = _normal_bf16(rng, (T, cfg.d), 1.0)
    n_users = (T + 127) // 128
    zipf = 1.0 / np.arange(1, cfg.M + 1)
    zipf /= zipf.sum()
    perm = rng.permutation(cfg.M)
    a_i = perm[rng.choice(cfg.M, size=n_users, p=zipf)]
    s = np.repeat(a_i, 128)[:T].astype(np.uint8)
    return dict(
        h=h,
        s=s,
        Dhat=np.zeros(T, dtype=np.float32),
        Dbar=np.full(T, cfg.budget, dtype=np.float32),
        pJ=np.full(T, cfg.p_J, dtype=np.float32),
        alive=np.ones(T, dtype=np.uint8),
        last_exec=np.zeros(T, dtype=np.uint8),
        xi_last=np.full(T, -1.0, dtype=np.float32),
        exit_layer=np.full(T, cfg.N, dtype=np.int16),
    )


def exit_profile(cfg: WorkloadConfig) -> np.ndarray:
    """Target fraction of all tokens that exit at each layer (sums to exit_target)."""
    N = cfg.N
    w = np.zeros(N)
    if cfg.exit_target <= 0 or N < 2:
        return w
    ls = np.arange(N, dtype=np.float64)
    if cfg.exit_peak is None:
        w[1:] = 1.0
    else:
        w = np.exp(-0.5 * ((ls - cfg.exit_peak) / cfg.exit_width) ** 2)
        w[0] = 0.0
    return w / w.sum() * cfg.exit_target
