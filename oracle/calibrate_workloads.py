"""Write paper_2608_00573_gb300/workload_calib.json (skip thresholds, exit biases).

Stand-in for the offline threshold calibration of Sec. IV-B (Eq. 24-25) on the
synthetic workloads.  The exit head's class-0 bias is set per layer so that the
share of tokens whose confidence reaches p_J follows the target exit profile;
then theta_l is the importance quantile q (the same q for every layer) found
by bisection so that an oracle decisions-only pilot over all layers skips the
target share of live layer-tokens.  Only the oracle computes router outputs,
exit-head logits and decisions here; the sample is the first tokens of the
seeded input.

    python oracle/calibrate_workloads.py            # all workloads
"""
from __future__ import annotations

import json
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

from oracle import oracle as O  # noqa: E402
from paper_2608_00573_gb300 import workload as W  # noqa: E402

SAMPLE = 1024
PILOT = 512


def calibrate(name: str) -> dict:
    cfg = W.CONFIGS[name]
    small = W.make_small_weights(cfg, calib=None)
    tables = W.make_tables(cfg, small["W_r"], calib=None)
    om = O.OracleModel(cfg, tables, small)
    tok = W.make_tokens(cfg, T=max(cfg.T, SAMPLE))
    h = tok["h"][:SAMPLE]
    Is = [np.array([O.router(om, l, h[t])[4] for t in range(len(h))], dtype=np.float64)
          for l in range(cfg.N)]
    # Exit: target share of the still-alive tokens at layer l with xi >= p_J.
    prof = W.exit_profile(cfg)
    alive = 1.0
    bias = [-30.0] * cfg.N
    logit_p = np.log(cfg.p_J / (1.0 - cfg.p_J))
    for l in range(1, cfg.N):
        target = prof[l] / max(alive, 1e-9) / max(1.0 - cfg.skip_target, 0.5)
        alive -= prof[l]
        if target <= 1e-6:
            continue
        target = min(target, 0.95)
        # Head l-1 logits with zero class-0 bias.
        Wx = small["W_x"][l - 1]
        X = np.stack([_head_logits(om, Wx, h[t]) for t in range(len(h))])   # [S, C]

        def share(b):
            Y = X.copy()
            Y[:, 0] += b
            if cfg.C == 1:
                return float(np.mean(Y[:, 0] >= logit_p))
            m = Y.max(axis=1, keepdims=True)
            xi = 1.0 / np.exp(Y - m).sum(axis=1)
            return float(np.mean(xi >= cfg.p_J))

        lo, hi = -60.0, 60.0
        for _ in range(60):
            mid = 0.5 * (lo + hi)
            if share(mid) < target:
                lo = mid
            else:
                hi = mid
        bias[l - 1] = float(hi)
    small_b = dict(small)
    small_b["b_x"] = small["b_x"].copy()
    small_b["b_x"][:, 0] = np.asarray(bias, dtype=np.float32)
    pilot = {k: v[:PILOT] for k, v in tok.items()}

    def skip_share(q):
        tab = dict(tables)
        tab["theta"] = np.array([np.quantile(I, q) for I in Is], dtype=np.float32)
        kappa = max(cfg.skip_target * cfg.N, 1.0)
        tab["eps"] = np.full(cfg.N, cfg.budget / kappa, dtype=np.float32)
        tab["lam"] = (tab["eps"] / np.maximum(tab["theta"], 1e-6)).astype(np.float32)
        pm = O.OracleModel(cfg, tab, small_b, None)
        hh = pilot["h"]
        st = {k: v for k, v in pilot.items() if k != "h"}
        skipped = live = 0
        for l in range(cfg.N):
            hh, st, out = O.layer_step(pm, l, hh, st, row_mask=np.zeros(len(hh), np.uint8))
            a = out["action"]
            skipped += int((a == O.A_SKIP).sum())
            live += int((a != O.A_DEAD).sum())
        return skipped / max(live, 1), tab["theta"]

    q = 0.0
    theta = [-1.0] * cfg.N
    achieved = 0.0
    if cfg.skip_target > 0:
        lo, hi = 0.0, 1.0
        for _ in range(9):
            mid = 0.5 * (lo + hi)
            sh, th = skip_share(mid)
            if sh < cfg.skip_target:
                lo = mid
            else:
                hi = mid
        q = hi
        achieved, th = skip_share(q)
        theta = [float(x) for x in th]
    return {"theta": theta, "exit_bias": bias, "sample_tokens": SAMPLE, "pilot_tokens": PILOT,
            "skip_quantile": q, "pilot_skip_share": achieved}


def _head_logits(om, Wx, h_row):
    import ctypes as C
    cfg = om.cfg
    out = np.zeros(cfg.C, np.float32)
    wx = np.ascontiguousarray(Wx, dtype=np.uint16)
    bx = np.zeros(cfg.C, np.float32)
    hr = np.ascontiguousarray(h_row, dtype=np.uint16)
    O.lib().or_exit_conf(C.byref(om.m), wx.ctypes.data, bx.ctypes.data, hr.ctypes.data,
                         int(cfg.norm), out.ctypes.data)
    return out.astype(np.float64)


def main(names=None):
    names = names or list(W.CONFIGS)
    data = {}
    if os.path.exists(W.CALIB_PATH):
        with open(W.CALIB_PATH) as fh:
            data = json.load(fh)
    for n in names:
        data[n] = calibrate(n)
        print(n, "theta[0..3]", [round(x, 4) for x in data[n]["theta"][:4]],
              "exit_bias", [round(x, 2) for x in data[n]["exit_bias"]])
    with open(W.CALIB_PATH, "w") as fh:
        json.dump(data, fh, indent=1)


if __name__ == "__main__":
    main(sys.argv[1:] or None)
