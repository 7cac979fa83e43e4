"""Write paper_2608_00573_gb300/workload_calib.json (skip thresholds, exit biases).

Stand-in for the offline threshold calibration of Sec. IV-B (Eq. 24-25) on the
synthetic workloads: theta_l is the importance quantile at which about the
target share of layer-tokens is admitted to skip, and the exit head's class-0
bias is set per layer so that the share of tokens whose confidence reaches p_J
follows the target exit profile.  Only the oracle computes router outputs and
exit-head logits here; the sample is the first tokens of the seeded input.

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
# Share of layer-tokens whose execute candidates are all remote on these
# placements (2-4 replicas of 10 servers, plus substitutes); skip admission by
# importance is scaled by its inverse.
REMOTE_SHARE = 0.5


def calibrate(name: str) -> dict:
    cfg = W.CONFIGS[name]
    small = W.make_small_weights(cfg, calib=None)
    tables = W.make_tables(cfg, small["W_r"], calib=None)
    om = O.OracleModel(cfg, tables, small)
    tok = W.make_tokens(cfg, T=max(cfg.T, SAMPLE))
    h = tok["h"][:SAMPLE]
    q = min(1.0, cfg.skip_target / REMOTE_SHARE)
    theta = []
    for l in range(cfg.N):
        I = np.array([O.router(om, l, h[t])[4] for t in range(len(h))], dtype=np.float64)
        theta.append(float(np.quantile(I, q)) if q > 0 else -1.0)
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
    return {"theta": theta, "exit_bias": bias, "sample_tokens": SAMPLE, "skip_quantile": q}


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
