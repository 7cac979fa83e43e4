"""ctypes binding of include/trimmoe.h (argument marshalling only).

Every step of the layer runs in the CUDA library; this module only converts
torch tensors / numpy arrays into the C structs and calls the entry points.
It raises if the compiled library is missing: there is no fallback path.
"""
from __future__ import annotations

import ctypes as C
import os
import threading
from typing import Optional

import numpy as np

from . import workload as W

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "_build", "libtrimmoe.so")

TRIMMOE_OK = 0
STATUS_NAMES = {0: "OK", -1: "ERR_ARG", -2: "ERR_UNSUPPORTED", -3: "ERR_OOM", -4: "ERR_CUDA",
                -5: "ERR_COVERAGE", -6: "ERR_DEVICE_TIMEOUT"}
EXEC, SKIP, EXIT, DEAD = 0, 1, 2, 3


class TrimmoeError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


class trimmoe_config(C.Structure):
    _fields_ = [(n, C.c_int) for n in ("N", "d", "E", "k", "F", "F_sh", "C", "M", "H", "act",
                                       "renorm_topk", "n_sub", "T_max")] + \
               [(n, C.c_float) for n in ("omega_T", "omega_D", "d_ref_ms", "phi_beta")] + \
               [("profile", C.c_int), ("norm_eps", C.c_float), ("n_centroids", C.c_int)] + \
               [(n, C.c_int) for n in ("attn_heads", "attn_kv_heads", "head_dim", "attn_seq")] + \
               [("rope_theta", C.c_float), ("graphs", C.c_int)]


class trimmoe_weights(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in ("W_r", "b_r", "W_x", "b_x", "W13", "W2", "W13_sh", "W2_sh",
                                          "W_norm", "centroids", "W_attn_norm", "W_qkv", "W_o")]


class trimmoe_tables(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in ("place", "sim", "sub_thresh", "trans_ms", "comp_ms", "P",
                                          "theta", "lambda_", "eps", "centroid_exit")]


class trimmoe_tokens(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in ("hidden", "s", "Dhat", "Dbar", "pJ", "alive", "last_exec",
                                          "xi_last", "exit_layer")]


class trimmoe_layer_out(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in ("topk_idx", "topk_g", "I", "xi", "action", "exp_sel",
                                          "srv_sel", "perm", "group_off", "lhat", "h_attn")]


class trimmoe_stats_t(C.Structure):
    _fields_ = [(n, C.c_uint64) for n in ("layer_tokens", "exec_tokens", "skipped", "exited",
                                          "pairs_local_exact", "pairs_local_sub", "pairs_remote_exact",
                                          "pairs_remote_sub", "shared_rows")] + \
               [("delay_ms", C.c_double), ("remote_hops", C.c_double), ("max_budget_ratio", C.c_float),
                ("device_error", C.c_int), ("launches", C.c_uint64), ("layer_calls", C.c_uint64),
                ("gemm_flops", C.c_double)] + \
               [(n, C.c_double) for n in ("ms_decide", "ms_compact", "ms_gather", "ms_gemm_up",
                                          "ms_gemm_down", "ms_combine")] + \
               [("n_gemm_up", C.c_uint64), ("n_gemm_down", C.c_uint64),
                ("flops_gemm_up", C.c_double), ("flops_gemm_down", C.c_double), ("ms_router", C.c_double),
                ("bytes_gemm_up", C.c_double), ("bytes_gemm_down", C.c_double),
                ("lookahead_shared", C.c_uint64),
                ("ms_attn", C.c_double), ("ms_attn_gemm", C.c_double), ("flops_attn", C.c_double),
                ("flops_attn_gemm", C.c_double), ("pairs_executed", C.c_uint64),
                ("bytes_expert_weights", C.c_double)]

    def as_dict(self):
        return {n: getattr(self, n) for n, _ in self._fields_}


class trimmoe_feedback_cfg(C.Structure):
    _fields_ = [("user_size", C.c_int), ("eta", C.c_float), ("p_min", C.c_float), ("kappa", C.c_float)]


class trimmoe_feedback_out(C.Structure):
    _fields_ = [("omega_T", C.c_float), ("omega_D", C.c_float), ("T_norm", C.c_double), ("D_util", C.c_double),
                ("users_updated", C.c_int), ("window_delay_ms", C.c_double), ("window_ref_slots", C.c_double)]

    def as_dict(self):
        return {n: getattr(self, n) for n, _ in self._fields_}


class trimmoe_calibration_t(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in ("trans", "alive", "resid", "act", "above", "P", "pi", "sigma",
                                          "act_freq", "lambda_", "rho")]


EXPORTS = ("trimmoe_create", "trimmoe_layer_step", "trimmoe_forward", "trimmoe_forward_host",
           "trimmoe_stats", "trimmoe_reset_stats", "trimmoe_last_error", "trimmoe_destroy",
           "trimmoe_compact_noalloc", "trimmoe_feedback", "trimmoe_calibration_begin",
           "trimmoe_calibration_end", "trimmoe_replicate", "trimmoe_watchdog_selftest")

_lib = None
_lock = threading.Lock()


def lib():
    """Load the CUDA library (raises if it has not been built)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                                   "`python -m paper_2608_00573_gb300.build`")
            L = C.CDLL(LIB_PATH)
            vp, i = C.c_void_p, C.c_int
            L.trimmoe_create.argtypes = [vp, vp, vp, C.POINTER(vp)]
            L.trimmoe_create.restype = i
            L.trimmoe_layer_step.argtypes = [vp, i, i, vp, vp, vp]
            L.trimmoe_layer_step.restype = i
            L.trimmoe_forward.argtypes = [vp, i, vp, vp]
            L.trimmoe_forward.restype = i
            L.trimmoe_forward_host.argtypes = [vp, i, vp, vp]
            L.trimmoe_forward_host.restype = i
            L.trimmoe_stats.argtypes = [vp, vp]
            L.trimmoe_stats.restype = i
            L.trimmoe_reset_stats.argtypes = [vp]
            L.trimmoe_reset_stats.restype = i
            L.trimmoe_watchdog_selftest.argtypes = [vp, i, vp]
            L.trimmoe_watchdog_selftest.restype = i
            L.trimmoe_last_error.argtypes = [vp]
            L.trimmoe_last_error.restype = C.c_char_p
            L.trimmoe_destroy.argtypes = [vp]
            L.trimmoe_destroy.restype = None
            L.trimmoe_compact_noalloc.argtypes = [vp, vp, i, i, i, i, vp, vp, vp, vp, vp]
            L.trimmoe_feedback.argtypes = [vp, vp, i, vp, vp, vp]
            L.trimmoe_feedback.restype = i
            L.trimmoe_calibration_begin.argtypes = [vp]
            L.trimmoe_calibration_begin.restype = i
            L.trimmoe_calibration_end.argtypes = [vp, C.c_longlong, vp]
            L.trimmoe_calibration_end.restype = i
            L.trimmoe_replicate.argtypes = [i, i, i, vp, vp, vp, vp, vp, vp, vp]
            L.trimmoe_replicate.restype = i
            L.trimmoe_compact_noalloc.restype = i
            _lib = L
    return _lib


def _check(rc, handle=None):
    if rc != TRIMMOE_OK:
        msg = lib().trimmoe_last_error(handle)
        raise TrimmoeError(rc, msg.decode() if msg else "")


# ----------------------------------------------------------- thin wrappers

def trimmoe_create(cfg: trimmoe_config, w: trimmoe_weights, tab: trimmoe_tables) -> C.c_void_p:
    h = C.c_void_p()
    _check(lib().trimmoe_create(C.byref(cfg), C.byref(w), C.byref(tab), C.byref(h)))
    return h


def trimmoe_layer_step(h, layer: int, T: int, tok: trimmoe_tokens, out: Optional[trimmoe_layer_out],
                       stream: int = 0):
    _check(lib().trimmoe_layer_step(h, layer, T, C.byref(tok), C.byref(out) if out is not None else None,
                                    C.c_void_p(stream)), h)


def trimmoe_forward(h, T: int, tok: trimmoe_tokens, stream: int = 0):
    _check(lib().trimmoe_forward(h, T, C.byref(tok), C.c_void_p(stream)), h)


def trimmoe_forward_host(h, T: int, tok: trimmoe_tokens, stream: int = 0):
    _check(lib().trimmoe_forward_host(h, T, C.byref(tok), C.c_void_p(stream)), h)


def trimmoe_stats(h) -> dict:
    s = trimmoe_stats_t()
    rc = lib().trimmoe_stats(h, C.byref(s))
    d = s.as_dict()
    d["status"] = rc
    return d


def trimmoe_reset_stats(h):
    _check(lib().trimmoe_reset_stats(h), h)


def trimmoe_watchdog_selftest(h, timeout_us: int, stream: int = 0) -> int:
    """Run the bounded-wait self-check; returns the status code (DEVICE_TIMEOUT when the
    wait ran out as designed) instead of raising."""
    return lib().trimmoe_watchdog_selftest(h, timeout_us, C.c_void_p(stream))


def trimmoe_last_error(h=None) -> str:
    m = lib().trimmoe_last_error(h)
    return m.decode() if m else ""


def trimmoe_destroy(h):
    lib().trimmoe_destroy(h)


def trimmoe_feedback(h, fb: trimmoe_feedback_cfg, T: int, tok: trimmoe_tokens, stream: int = 0) -> dict:
    out = trimmoe_feedback_out()
    _check(lib().trimmoe_feedback(h, C.byref(fb), T, C.byref(tok), C.byref(out), C.c_void_p(stream)), h)
    return out.as_dict()


def trimmoe_calibration_begin(h):
    _check(lib().trimmoe_calibration_begin(h), h)


def trimmoe_calibration_end(h, T_cal: int, N: int, E: int, M: int) -> dict:
    """Counts and statistics of the offline stage as numpy arrays."""
    o = dict(trans=np.zeros((max(N - 1, 1), E, E), np.uint64), alive=np.zeros(N, np.uint64),
             resid=np.zeros((N, M), np.uint64), act=np.zeros((N, E), np.uint64), above=np.zeros((N, E), np.uint64),
             P=np.zeros((max(N - 1, 1), E, E), np.float32), pi=np.zeros(N, np.float32),
             sigma=np.zeros((N, E), np.float32), act_freq=np.zeros((N, E), np.float32),
             lam=np.zeros((N, E), np.float32), rho=np.zeros((N, M), np.float32))
    st = trimmoe_calibration_t(trans=_ptr(o["trans"]), alive=_ptr(o["alive"]), resid=_ptr(o["resid"]),
                               act=_ptr(o["act"]), above=_ptr(o["above"]), P=_ptr(o["P"]), pi=_ptr(o["pi"]),
                               sigma=_ptr(o["sigma"]), act_freq=_ptr(o["act_freq"]), lambda_=_ptr(o["lam"]),
                               rho=_ptr(o["rho"]))
    _check(lib().trimmoe_calibration_end(h, int(T_cal), C.byref(st)), h)
    return o


def trimmoe_replicate(lam, rho, trans, expert_bytes, capacity, place):
    """Greedy replication (Eq. 28) on a copy of place (host arrays); returns (place, added)."""
    N, E = place.shape
    M = trans.shape[0]
    pl = np.array(place, dtype=np.uint16, copy=True)
    arrs = [np.ascontiguousarray(a, dt) for a, dt in ((lam, np.float32), (rho, np.float32), (trans, np.float32),
                                                        (expert_bytes, np.float64), (capacity, np.float64))]
    added = C.c_int(0)
    _check(lib().trimmoe_replicate(N, E, M, *[_ptr(a) for a in arrs], _ptr(pl), C.byref(added)))
    return pl, added.value


def trimmoe_compact_noalloc(action, exp_sel, T: int, k: int, E: int, has_shared: int, perm, group_off,
                            pos_pair, pos_sh, stream: int = 0):
    """Compaction into caller-owned outputs with no device allocation (device tensors)."""
    _check(lib().trimmoe_compact_noalloc(_ptr(action), _ptr(exp_sel), T, k, E, has_shared, _ptr(perm),
                                         _ptr(group_off), _ptr(pos_pair), _ptr(pos_sh), C.c_void_p(stream)))


# ----------------------------------------------------------- engine

TOKEN_FIELDS = ("hidden", "s", "Dhat", "Dbar", "pJ", "alive", "last_exec", "xi_last", "exit_layer")


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, np.ndarray):
        return t.ctypes.data
    return t.data_ptr()


class Engine:
    """Owns a trimmoe handle plus the torch tensors it borrows."""

    def __init__(self, cfg: W.WorkloadConfig, tables: dict, small: dict, experts: dict, T_max: int,
                 device="cuda", profile=False, graphs: bool = False):
        import torch
        self.torch = torch
        self.cfg = cfg
        self.device = torch.device(device)
        dev = self.device

        def dt(a, dtype):
            if isinstance(a, torch.Tensor):
                return a.to(dev).contiguous()
            a = np.ascontiguousarray(a)
            if a.dtype == np.uint16:
                return torch.from_numpy(a.view(np.int16)).to(dev).view(torch.bfloat16).contiguous()
            return torch.from_numpy(a).to(dev, dtype=dtype).contiguous()

        self.w = {
            "W_r": dt(small["W_r"], torch.bfloat16), "b_r": dt(small["b_r"], torch.float32),
            "W_x": dt(small["W_x"], torch.bfloat16), "b_x": dt(small["b_x"], torch.float32),
            "W13": dt(experts["W13"], torch.bfloat16), "W2": dt(experts["W2"], torch.bfloat16),
            "W13_sh": dt(experts["W13_sh"], torch.bfloat16) if cfg.F_sh else None,
            "W2_sh": dt(experts["W2_sh"], torch.bfloat16) if cfg.F_sh else None,
            "W_norm": dt(small["W_norm"], torch.bfloat16) if small.get("W_norm") is not None else None,
            "centroids": dt(small["centroids"], torch.bfloat16) if cfg.n_centroids else None,
            "W_attn_norm": dt(small["W_attn_norm"], torch.bfloat16) if cfg.attn_heads else None,
            "W_qkv": dt(experts["W_qkv"], torch.bfloat16) if cfg.attn_heads else None,
            "W_o": dt(experts["W_o"], torch.bfloat16) if cfg.attn_heads else None,
        }
        self.tables = {k: np.ascontiguousarray(v) for k, v in tables.items() if k != "d_ref"}
        self.c_cfg = trimmoe_config(
            N=cfg.N, d=cfg.d, E=cfg.E, k=cfg.k, F=cfg.F, F_sh=cfg.F_sh, C=cfg.C, M=cfg.M, H=cfg.H,
            act=cfg.act, renorm_topk=cfg.renorm_topk, n_sub=cfg.n_sub, T_max=T_max,
            omega_T=cfg.omega_T, omega_D=cfg.omega_D, d_ref_ms=float(tables["d_ref"]),
            phi_beta=cfg.phi_beta, profile=int(profile), norm_eps=cfg.norm_eps,
            n_centroids=cfg.n_centroids, attn_heads=cfg.attn_heads, attn_kv_heads=cfg.attn_kv_heads,
            head_dim=cfg.head_dim, attn_seq=cfg.attn_seq, rope_theta=cfg.rope_theta, graphs=1 if graphs else 0)
        self.c_w = trimmoe_weights(**{k: _ptr(v) for k, v in self.w.items()})
        t = self.tables
        P = t["P"].astype(np.float32) if t["P"].size else None
        self._P = P
        self.c_tab = trimmoe_tables(
            place=_ptr(t["place"].astype(np.uint16)), sim=_ptr(t["sim"]), sub_thresh=_ptr(t["sub_thresh"]),
            trans_ms=_ptr(t["trans"]), comp_ms=_ptr(t["comp"]), P=_ptr(P), theta=_ptr(t["theta"]),
            lambda_=_ptr(t["lam"]), eps=_ptr(t["eps"]))
        self._keep_place = t["place"].astype(np.uint16)
        self.c_tab.place = _ptr(self._keep_place)
        if cfg.n_centroids:
            self._cexit = np.ascontiguousarray(small["centroid_exit"], dtype=np.float32)
            self.c_tab.centroid_exit = _ptr(self._cexit)
        self.T_max = T_max
        self.handle = trimmoe_create(self.c_cfg, self.c_w, self.c_tab)

    # token state ----------------------------------------------------------
    def tokens_to_device(self, tok: dict):
        torch = self.torch
        out = {}
        for k in TOKEN_FIELDS:
            a = tok["h" if k == "hidden" else k]
            if isinstance(a, torch.Tensor):
                out[k] = a.to(self.device).contiguous()
            else:
                a = np.ascontiguousarray(a)
                if k == "hidden":
                    out[k] = torch.from_numpy(a.view(np.int16)).to(self.device).view(torch.bfloat16)
                else:
                    out[k] = torch.from_numpy(a).to(self.device)
        return out

    @staticmethod
    def tokens_to_host(tok: dict) -> dict:
        import torch
        out = {}
        for k, v in tok.items():
            v = v.detach().cpu()
            if k == "hidden":
                out["h"] = v.view(torch.int16).numpy().view(np.uint16).copy()
            else:
                out[k] = v.numpy().copy()
        return out

    def c_tokens(self, tok: dict) -> trimmoe_tokens:
        return trimmoe_tokens(**{k: _ptr(tok[k]) for k in TOKEN_FIELDS})

    def alloc_layer_out(self, T: int) -> dict:
        torch = self.torch
        K, E, dev = self.cfg.k, self.cfg.E, self.device
        return dict(
            topk_idx=torch.empty(T * K, dtype=torch.int32, device=dev),
            topk_g=torch.empty(T * K, dtype=torch.float32, device=dev),
            I=torch.empty(T, dtype=torch.float32, device=dev),
            xi=torch.empty(T, dtype=torch.float32, device=dev),
            action=torch.empty(T, dtype=torch.uint8, device=dev),
            exp_sel=torch.empty(T * K, dtype=torch.uint8, device=dev),
            srv_sel=torch.empty(T * K, dtype=torch.uint8, device=dev),
            perm=torch.full((T * K + T,), -1, dtype=torch.int32, device=dev),
            group_off=torch.empty(E + 2, dtype=torch.int32, device=dev),
            lhat=torch.empty(T, dtype=torch.int16, device=dev),
            h_attn=(torch.empty((T, self.cfg.d), dtype=torch.bfloat16, device=dev) if self.cfg.attn_heads
                    else None))

    def stream_ptr(self, stream=None) -> int:
        torch = self.torch
        s = stream if stream is not None else torch.cuda.current_stream(self.device)
        return int(s.cuda_stream)

    def layer_step(self, layer: int, tok: dict, T: Optional[int] = None, out: Optional[dict] = None,
                   stream=None):
        T = tok["s"].shape[0] if T is None else T
        c_out = trimmoe_layer_out(**{k: _ptr(v) for k, v in out.items()}) if out is not None else None
        trimmoe_layer_step(self.handle, layer, T, self.c_tokens(tok), c_out, self.stream_ptr(stream))
        return out

    def forward(self, tok: dict, T: Optional[int] = None, stream=None):
        T = tok["s"].shape[0] if T is None else T
        trimmoe_forward(self.handle, T, self.c_tokens(tok), self.stream_ptr(stream))

    def forward_host(self, host_tok: dict, T: Optional[int] = None, stream=None):
        """host_tok: dict of pinned CPU torch tensors keyed by TOKEN_FIELDS."""
        T = host_tok["s"].shape[0] if T is None else T
        trimmoe_forward_host(self.handle, T, self.c_tokens(host_tok), self.stream_ptr(stream))

    def stats(self) -> dict:
        return trimmoe_stats(self.handle)

    def calibration_begin(self):
        trimmoe_calibration_begin(self.handle)

    def calibration_end(self, T_cal: int) -> dict:
        return trimmoe_calibration_end(self.handle, T_cal, self.cfg.N, self.cfg.E, self.cfg.M)

    def feedback(self, tok: dict, user_size: int, eta: float, p_min: float, kappa: float,
                 T: Optional[int] = None, stream=None) -> dict:
        """Eq. (37) / (43) at the end of an observation window (updates tok['pJ'] in place)."""
        T = tok["s"].shape[0] if T is None else T
        fb = trimmoe_feedback_cfg(user_size=user_size, eta=eta, p_min=p_min, kappa=kappa)
        return trimmoe_feedback(self.handle, fb, T, self.c_tokens(tok), self.stream_ptr(stream))

    def reset_stats(self):
        trimmoe_reset_stats(self.handle)

    def close(self):
        if getattr(self, "handle", None):
            trimmoe_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
