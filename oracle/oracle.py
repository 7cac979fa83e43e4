"""ctypes wrapper of the CPU oracle (test infrastructure only).

Only the tests, the smoke check and the benchmark's CPU-baseline leg load this
module.  It compiles ``trimmoe_oracle.cpp`` with gcc (``-ffp-contract=off``,
OpenMP) into ``oracle/_build/liboracle.so`` and exposes numpy-level helpers.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "trimmoe_oracle.cpp")
BUILD_DIR = os.path.join(HERE, "_build")
LIB_PATH = os.path.join(BUILD_DIR, "liboracle.so")

A_EXEC, A_SKIP, A_EXIT, A_DEAD = 0, 1, 2, 3

_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    os.makedirs(BUILD_DIR, exist_ok=True)
    if force or not os.path.exists(LIB_PATH) or os.path.getmtime(LIB_PATH) < os.path.getmtime(SRC):
        tmp = LIB_PATH + f".{os.getpid()}.tmp"
        cmd = ["g++", "-O2", "-std=c++17", "-fPIC", "-shared", "-ffp-contract=off", "-fno-fast-math",
               "-fopenmp", "-o", tmp, SRC]
        subprocess.check_call(cmd)
        os.replace(tmp, LIB_PATH)
    return LIB_PATH


class OrModel(C.Structure):
    _fields_ = [(n, C.c_int) for n in
                ("N", "d", "E", "k", "F", "F_sh", "C", "M", "H", "act", "renorm_topk", "n_sub")] + \
               [(n, C.c_float) for n in ("omega_T", "omega_D", "d_ref", "phi_beta", "norm_eps")] + [
        ("place", C.c_void_p), ("sim", C.c_void_p), ("sub_thresh", C.c_void_p),
        ("trans", C.c_void_p), ("comp", C.c_void_p), ("P", C.c_void_p), ("theta", C.c_void_p),
        ("lambda_", C.c_void_p), ("eps", C.c_void_p), ("n_centroids", C.c_int),
        ("attn_heads", C.c_int), ("attn_kv_heads", C.c_int), ("head_dim", C.c_int), ("attn_seq", C.c_int),
        ("rope_theta", C.c_float)]


class OrLayerWeights(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in
                ("W_r", "b_r", "W_x_prev", "b_x_prev", "W13", "W2", "W13_sh", "W2_sh", "W_norm",
                 "centroids", "centroid_exit", "W_attn_norm", "W_qkv", "W_o")]


class OrTokens(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in
                ("s", "Dhat", "Dbar", "pJ", "alive", "last_exec", "xi_last", "exit_layer")]


class OrLayerOut(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in
                ("topk_idx", "topk_g", "I", "xi", "action", "exp_sel", "srv_sel", "perm",
                 "group_off", "near", "Gamma", "tot_exec", "tot_skip", "lhat")]


class OrDecision(C.Structure):
    _fields_ = [("topk", C.c_int * 16), ("g", C.c_float * 16)] + \
               [(n, C.c_float) for n in ("I", "xi", "Gamma", "tot_exec", "tot_skip", "Lambda")] + \
               [(n, C.c_int) for n in ("action", "skip_ok", "exit_ok")] + \
               [("exp_sel", C.c_int * 16), ("srv_sel", C.c_int * 16), ("Q_sel", C.c_float * 16),
                ("f_sel", C.c_float * 16), ("Dhat_new", C.c_float), ("s_new", C.c_int), ("near", C.c_int),
                ("Lhat", C.c_int)]


class OrFeedbackCfg(C.Structure):
    _fields_ = [("user_size", C.c_int), ("eta", C.c_float), ("p_min", C.c_float), ("kappa", C.c_float)]


class OrFeedbackOut(C.Structure):
    _fields_ = [("omega_T", C.c_float), ("omega_D", C.c_float), ("T_norm", C.c_double),
                ("D_util", C.c_double), ("users_updated", C.c_int)]


def lib():
    global _lib
    with _lock:
        if _lib is None:
            L = C.CDLL(build())
            vp, i, f = C.c_void_p, C.c_int, C.c_float
            L.or_router.argtypes = [vp, vp, vp, vp, vp, vp, vp, vp, vp, vp]
            L.or_exit_conf.argtypes = [vp, vp, vp, vp, i, vp]
            L.or_rms_factor.argtypes = [vp, i, f]
            L.or_rms_factor.restype = C.c_double
            L.or_exit_conf.restype = f
            L.or_sub_loss.argtypes = [vp, i, i, i]
            L.or_sub_loss.restype = f
            L.or_candidates.argtypes = [vp, i, i, vp, vp, vp, i]
            L.or_candidates.restype = i
            L.or_exec_cost.argtypes = [vp, i, i, i, f, f]
            L.or_exec_cost.restype = f
            L.or_lookahead_table.argtypes = [vp, i, f, f, vp]
            L.or_lookahead_table_capped.argtypes = [vp, i, f, f, i, vp]
            L.or_predict_exit.argtypes = [vp, vp, vp, vp, vp, vp]
            L.or_predict_exit.restype = i
            L.or_phi_naive.argtypes = [vp, i, i, i, i, f, f]
            L.or_phi_naive.restype = f
            L.or_decide_given.argtypes = [vp, i, vp, vp, f, f, i, f, f, f, i, vp]
            L.or_decide_token.argtypes = [vp, vp, i, vp, i, f, f, f, i, vp, vp]
            L.or_ffn_row.argtypes = [i, i, i, vp, vp, vp, vp]
            L.or_layer_step.argtypes = [vp, vp, i, i, vp, vp, vp, vp, i]
            L.or_layer_step.restype = i
            L.or_layer_step_block.argtypes = [vp, vp, i, i, vp, vp, vp, vp, vp, i]
            L.or_layer_step_block.restype = i
            L.or_attention.argtypes = [vp, vp, i, vp, vp, vp, vp, i]
            L.or_attention.restype = i
            L.or_rope.argtypes = [vp, i, i, C.c_double, vp]
            L.or_forward.argtypes = [vp, vp, i, vp, vp, i]
            L.or_forward.restype = i
            L.or_max_threads.restype = i
            L.or_feedback.argtypes = [vp, i, i, vp, vp, vp, vp, vp, vp, C.c_double, C.c_double, f, f, vp]
            L.or_feedback.restype = i
            L.or_calib_accumulate.argtypes = [vp, i, i, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp]
            L.or_calib_finalize.argtypes = [vp, C.c_longlong, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp]
            L.or_replicate.argtypes = [vp, vp, vp, vp, vp, vp]
            L.or_replicate.restype = i
            _lib = L
    return _lib


def _p(a):
    return None if a is None else a.ctypes.data


class OracleModel:
    """Holds the numpy arrays alive and the ctypes model struct."""

    def __init__(self, cfg, tables, small, experts=None):
        self.cfg = cfg
        self.keep = {}
        def keep(name, a, dt):
            a = np.ascontiguousarray(a, dtype=dt)
            self.keep[name] = a
            return a
        t = tables
        self.m = OrModel(
            N=cfg.N, d=cfg.d, E=cfg.E, k=cfg.k, F=cfg.F, F_sh=cfg.F_sh, C=cfg.C, M=cfg.M, H=cfg.H,
            act=cfg.act, renorm_topk=cfg.renorm_topk, n_sub=cfg.n_sub,
            omega_T=cfg.omega_T, omega_D=cfg.omega_D, d_ref=t["d_ref"], phi_beta=cfg.phi_beta,
            norm_eps=cfg.norm_eps,
            place=_p(keep("place", t["place"], np.uint16)), sim=_p(keep("sim", t["sim"], np.float32)),
            sub_thresh=_p(keep("sub_thresh", t["sub_thresh"], np.float32)),
            trans=_p(keep("trans", t["trans"], np.float32)), comp=_p(keep("comp", t["comp"], np.float32)),
            P=_p(keep("P", t["P"] if t["P"].size else np.zeros((1, cfg.E, cfg.E)), np.float32)),
            theta=_p(keep("theta", t["theta"], np.float32)), lambda_=_p(keep("lam", t["lam"], np.float32)),
            eps=_p(keep("eps", t["eps"], np.float32)), n_centroids=cfg.n_centroids,
            attn_heads=cfg.attn_heads, attn_kv_heads=cfg.attn_kv_heads, head_dim=cfg.head_dim,
            attn_seq=cfg.attn_seq, rope_theta=cfg.rope_theta)
        self.small = {k: (None if v is None else np.ascontiguousarray(v)) for k, v in small.items()}
        self.experts = experts   # dict of numpy arrays (bf16 bits) per layer or full, or None

    def layer_weights(self, l, experts_l=None):
        """experts_l: dict with W13, W2 (and W13_sh, W2_sh) for layer l (uint16 arrays)."""
        s = self.small
        if experts_l is None:
            e = self.experts or {}
            experts_l = {k: e[k][l] for k in e}
        ex = {k: np.ascontiguousarray(v, dtype=np.uint16) for k, v in experts_l.items()}
        br = np.ascontiguousarray(s["b_r"][l], dtype=np.float32)
        wr = np.ascontiguousarray(s["W_r"][l], dtype=np.uint16)
        wx = np.ascontiguousarray(s["W_x"][l - 1], dtype=np.uint16) if l > 0 else None
        bx = np.ascontiguousarray(s["b_x"][l - 1], dtype=np.float32) if l > 0 else None
        wn = np.ascontiguousarray(s["W_norm"][l], dtype=np.uint16) if s.get("W_norm") is not None else None
        cc = ce = None
        if self.cfg.n_centroids and s.get("centroids") is not None:
            cc = np.ascontiguousarray(s["centroids"][l], dtype=np.uint16)
            ce = np.ascontiguousarray(s["centroid_exit"][l], dtype=np.float32)
        an = None
        if self.cfg.attn_heads and s.get("W_attn_norm") is not None:
            an = np.ascontiguousarray(s["W_attn_norm"][l], dtype=np.uint16)
        lw = OrLayerWeights(W_r=_p(wr), b_r=_p(br), W_x_prev=_p(wx), b_x_prev=_p(bx),
                            W13=_p(ex.get("W13")), W2=_p(ex.get("W2")),
                            W13_sh=_p(ex.get("W13_sh")), W2_sh=_p(ex.get("W2_sh")), W_norm=_p(wn),
                            centroids=_p(cc), centroid_exit=_p(ce), W_attn_norm=_p(an),
                            W_qkv=_p(ex.get("W_qkv")), W_o=_p(ex.get("W_o")))
        lw._keep = (wr, br, wx, bx, ex, wn, cc, ce, an)
        return lw


def tokens_struct(tok):
    arrs = {
        "s": np.ascontiguousarray(tok["s"], dtype=np.uint8),
        "Dhat": np.ascontiguousarray(tok["Dhat"], dtype=np.float32),
        "Dbar": np.ascontiguousarray(tok["Dbar"], dtype=np.float32),
        "pJ": np.ascontiguousarray(tok["pJ"], dtype=np.float32),
        "alive": np.ascontiguousarray(tok["alive"], dtype=np.uint8),
        "last_exec": np.ascontiguousarray(tok["last_exec"], dtype=np.uint8),
        "xi_last": np.ascontiguousarray(tok["xi_last"], dtype=np.float32),
        "exit_layer": np.ascontiguousarray(tok["exit_layer"], dtype=np.int16),
    }
    st = OrTokens(**{k: _p(v) for k, v in arrs.items()})
    return st, arrs


def alloc_layer_out(T, cfg):
    K, E = cfg.k, cfg.E
    o = dict(
        topk_idx=np.zeros(T * K, np.int32), topk_g=np.zeros(T * K, np.float32),
        I=np.zeros(T, np.float32), xi=np.zeros(T, np.float32), action=np.zeros(T, np.uint8),
        exp_sel=np.zeros(T * K, np.uint8), srv_sel=np.zeros(T * K, np.uint8),
        perm=np.full(T * K + T, -1, np.int32), group_off=np.zeros(E + 2, np.int32),
        near=np.zeros(T, np.uint8), Gamma=np.zeros(T, np.float32), tot_exec=np.zeros(T, np.float32),
        tot_skip=np.zeros(T, np.float32), lhat=np.zeros(T, np.int16))
    return OrLayerOut(**{k: _p(v) for k, v in o.items()}), o


def layer_step(om: OracleModel, l, h, tok, experts_l=None, row_mask=None, nthreads=0, h_mid=None):
    """Run one layer; returns (h_out, tokens_out, outputs). Inputs are not modified.
    With an attention sublayer, h_mid (bf16 bits [T][d]) supplies the state after
    attention; None computes it."""
    T = h.shape[0]
    h = np.array(h, dtype=np.uint16, copy=True, order="C")
    st, arrs = tokens_struct({k: np.array(v, copy=True) for k, v in tok.items()})
    out_s, out = alloc_layer_out(T, om.cfg)
    lw = om.layer_weights(l, experts_l)
    rm = None if row_mask is None else np.ascontiguousarray(row_mask, dtype=np.uint8)
    hm = None if h_mid is None else np.ascontiguousarray(h_mid, dtype=np.uint16)
    rc = lib().or_layer_step_block(C.byref(om.m), C.byref(lw), l, T, _p(h), _p(hm), C.byref(st),
                                   C.byref(out_s), _p(rm), nthreads)
    if rc:
        raise RuntimeError(f"or_layer_step failed: {rc}")
    return h, arrs, out


def attention(om: OracleModel, l, h, alive, experts_l=None, row_mask=None, nthreads=0):
    """State after the attention sublayer of layer l (bf16 bits [T][d]); rows of
    tokens that are not live or not in row_mask are copies of h."""
    T = h.shape[0]
    h = np.ascontiguousarray(h, dtype=np.uint16)
    out = np.zeros_like(h)
    lw = om.layer_weights(l, experts_l)
    al = np.ascontiguousarray(alive, dtype=np.uint8)
    rm = None if row_mask is None else np.ascontiguousarray(row_mask, dtype=np.uint8)
    rc = lib().or_attention(C.byref(om.m), C.byref(lw), T, _p(h), _p(al), _p(rm), _p(out), nthreads)
    if rc:
        raise RuntimeError(f"or_attention failed: {rc}")
    return out


def rope(x, pos, theta):
    """Rotary embedding of one head vector (float64)."""
    x = np.ascontiguousarray(x, dtype=np.float64)
    y = np.zeros_like(x)
    lib().or_rope(_p(x), x.size, int(pos), float(theta), _p(y))
    return y


def forward(om: OracleModel, h, tok, nthreads=0):
    T = h.shape[0]
    h = np.array(h, dtype=np.uint16, copy=True, order="C")
    st, arrs = tokens_struct({k: np.array(v, copy=True) for k, v in tok.items()})
    lws = (OrLayerWeights * om.cfg.N)()
    keep = []
    for l in range(om.cfg.N):
        lw = om.layer_weights(l)
        keep.append(lw)
        lws[l] = lw
    rc = lib().or_forward(C.byref(om.m), lws, T, _p(h), C.byref(st), nthreads)
    if rc:
        raise RuntimeError(f"or_forward failed: {rc}")
    return h, arrs


def router(om: OracleModel, l, h_row):
    cfg = om.cfg
    z = np.zeros(cfg.E, np.float32); p = np.zeros(cfg.E, np.float32)
    topk = np.zeros(16, np.int32); g = np.zeros(16, np.float32); I = np.zeros(1, np.float32)
    wr = np.ascontiguousarray(om.small["W_r"][l], dtype=np.uint16)
    br = np.ascontiguousarray(om.small["b_r"][l], dtype=np.float32)
    wn = om.small.get("W_norm")
    wn = None if wn is None else np.ascontiguousarray(wn[l], dtype=np.uint16)
    hr = np.ascontiguousarray(h_row, dtype=np.uint16)
    lib().or_router(C.byref(om.m), _p(wr), _p(br), _p(wn), _p(hr), _p(z), _p(p), _p(topk), _p(g), _p(I))
    return z, p, topk[:cfg.k].copy(), g[:cfg.k].copy(), float(I[0])


def exit_conf(om: OracleModel, W_x_l, b_x_l, h_row, normalise=None):
    wx = np.ascontiguousarray(W_x_l, dtype=np.uint16)
    bx = np.ascontiguousarray(b_x_l, dtype=np.float32)
    hr = np.ascontiguousarray(h_row, dtype=np.uint16)
    if normalise is None:
        normalise = om.small.get("W_norm") is not None
    return float(lib().or_exit_conf(C.byref(om.m), _p(wx), _p(bx), _p(hr), int(normalise), None))


def rms_factor(om: OracleModel, h_row):
    hr = np.ascontiguousarray(h_row, dtype=np.uint16)
    return float(lib().or_rms_factor(_p(hr), om.cfg.d, C.c_float(om.cfg.norm_eps)))


def candidates(om: OracleModel, l, r):
    cap = om.cfg.M * om.cfg.E
    cm = np.zeros(cap, np.int32); ck = np.zeros(cap, np.int32); cQ = np.zeros(cap, np.float32)
    n = lib().or_candidates(C.byref(om.m), l, r, _p(cm), _p(ck), _p(cQ), cap)
    return [(int(cm[i]), int(ck[i]), float(cQ[i])) for i in range(n)]


def exec_cost(om, l, s, m, Q, Dbar):
    return float(lib().or_exec_cost(C.byref(om.m), l, s, m, C.c_float(Q), C.c_float(Dbar)))


def lookahead_table(om, l, R, Dbar):
    out = np.zeros(om.cfg.M * om.cfg.E, np.float32)
    lib().or_lookahead_table(C.byref(om.m), l, C.c_float(R), C.c_float(Dbar), _p(out))
    return out.reshape(om.cfg.M, om.cfg.E)


def lookahead_table_capped(om, l, R, Dbar, cap):
    out = np.zeros(om.cfg.M * om.cfg.E, np.float32)
    lib().or_lookahead_table_capped(C.byref(om.m), l, C.c_float(R), C.c_float(Dbar), cap, _p(out))
    return out.reshape(om.cfg.M, om.cfg.E)


def predict_exit(om, centroids_l, centroid_exit_l, h_row):
    c = np.ascontiguousarray(centroids_l, dtype=np.uint16)
    e = np.ascontiguousarray(centroid_exit_l, dtype=np.float32)
    hr = np.ascontiguousarray(h_row, dtype=np.uint16)
    best = np.zeros(1, np.float32); gap = np.zeros(1, np.float32)
    L = lib().or_predict_exit(C.byref(om.m), _p(c), _p(e), _p(hr), _p(best), _p(gap))
    return int(L), float(best[0]), float(gap[0])


def phi_naive(om, l, h, m, k, R, Dbar):
    return float(lib().or_phi_naive(C.byref(om.m), l, h, m, k, C.c_float(R), C.c_float(Dbar)))


def decide_given(om, l, topk, g, I, xi, s, Dhat, Dbar, pJ, last_exec):
    tk = np.zeros(16, np.int32); tk[:len(topk)] = topk
    gg = np.zeros(16, np.float32); gg[:len(g)] = g
    D = OrDecision()
    lib().or_decide_given(C.byref(om.m), l, _p(tk), _p(gg), C.c_float(I), C.c_float(xi), s,
                          C.c_float(Dhat), C.c_float(Dbar), C.c_float(pJ), last_exec, C.byref(D))
    return D


def ffn_row(d, F, act, W13_e, W2_e, x):
    y = np.zeros(d, np.uint16)
    w13 = np.ascontiguousarray(W13_e, dtype=np.uint16)
    w2 = np.ascontiguousarray(W2_e, dtype=np.uint16)
    xx = np.ascontiguousarray(x, dtype=np.uint16)
    lib().or_ffn_row(d, F, act, _p(w13), _p(w2), _p(xx), _p(y))
    return y


def max_threads():
    return int(lib().or_max_threads())


def feedback(tok, N, user_size, eta, p_min, kappa, delay_sum_ms, ref_slots, d_ref, omega_D):
    """Eq. (37) and (43) on host arrays; returns (new pJ, OrFeedbackOut)."""
    T = len(tok["pJ"])
    pJ = np.array(tok["pJ"], dtype=np.float32, copy=True)
    arr = {k: np.ascontiguousarray(tok[k], dtype=dt) for k, dt in
           (("alive", np.uint8), ("exit_layer", np.int16), ("xi_last", np.float32), ("Dhat", np.float32),
            ("Dbar", np.float32))}
    cfg = OrFeedbackCfg(user_size=user_size, eta=eta, p_min=p_min, kappa=kappa)
    out = OrFeedbackOut()
    rc = lib().or_feedback(C.byref(cfg), T, N, _p(pJ), _p(arr["alive"]), _p(arr["exit_layer"]), _p(arr["xi_last"]),
                           _p(arr["Dhat"]), _p(arr["Dbar"]), C.c_double(delay_sum_ms), C.c_double(ref_slots),
                           C.c_float(d_ref), C.c_float(omega_D), C.byref(out))
    if rc:
        raise RuntimeError("or_feedback failed")
    return pJ, out


class CalibCounts:
    """Calibration counters of the offline stage (host, uint64)."""

    def __init__(self, cfg):
        N, E, M = cfg.N, cfg.E, cfg.M
        self.cfg = cfg
        self.trans = np.zeros((max(N - 1, 1), E, E), np.uint64)
        self.alive = np.zeros(N, np.uint64)
        self.resid = np.zeros((N, M), np.uint64)
        self.act = np.zeros((N, E), np.uint64)
        self.above = np.zeros((N, E), np.uint64)

    def accumulate(self, om, l, out, s_before, prev_target):
        T = len(s_before)
        ti = np.ascontiguousarray(out["topk_idx"], np.int32)
        I = np.ascontiguousarray(out["I"], np.float32)
        a = np.ascontiguousarray(out["action"], np.uint8)
        sb = np.ascontiguousarray(s_before, np.uint8)
        lib().or_calib_accumulate(C.byref(om.m), l, T, _p(ti), _p(I), _p(a), _p(sb), _p(prev_target),
                                  _p(self.trans), _p(self.alive), _p(self.resid), _p(self.act), _p(self.above))

    def finalize(self, om, T_cal):
        cfg = self.cfg
        N, E, M = cfg.N, cfg.E, cfg.M
        out = dict(P=np.zeros((max(N - 1, 1), E, E), np.float32), pi=np.zeros(N, np.float32),
                   sigma=np.zeros((N, E), np.float32), act=np.zeros((N, E), np.float32),
                   lam=np.zeros((N, E), np.float32), rho=np.zeros((N, M), np.float32))
        lib().or_calib_finalize(C.byref(om.m), int(T_cal), _p(self.trans), _p(self.alive), _p(self.resid),
                                _p(self.act), _p(self.above), _p(out["P"]), _p(out["pi"]), _p(out["sigma"]),
                                _p(out["act"]), _p(out["lam"]), _p(out["rho"]))
        return out


def replicate(om, lam, rho, expert_bytes, capacity, place):
    """Greedy replication (Eq. 28) on a copy of place; returns (new place, replicas added)."""
    pl = np.array(place, dtype=np.uint16, copy=True)
    lam = np.ascontiguousarray(lam, np.float32)
    rho = np.ascontiguousarray(rho, np.float32)
    eb = np.ascontiguousarray(expert_bytes, np.float64)
    cap = np.ascontiguousarray(capacity, np.float64)
    n = lib().or_replicate(C.byref(om.m), _p(lam), _p(rho), _p(eb), _p(cap), _p(pl))
    return pl, int(n)
