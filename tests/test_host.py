"""Host-only checks of the C ABI library and of the benchmark's multi-rank logic."""
import ctypes as C
import os
import re

import numpy as np
import pytest

from paper_2608_00573_gb300 import binding as B
from paper_2608_00573_gb300 import build as BUILD
from paper_2608_00573_gb300 import workload as W
from tests.oracle_helpers import small_cfg

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    BUILD.build()
    return B.lib()


def declared_functions():
    with open(os.path.join(ROOT, "include", "trimmoe.h")) as fh:
        src = fh.read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(trimmoe_[a-z_]+)\s*\(", src)))


def test_library_exports_every_declared_symbol(lib):
    names = declared_functions()
    assert set(B.EXPORTS) <= set(names)
    for n in names:
        assert hasattr(lib, n), n


def test_header_struct_sizes_match_binding():
    """The ctypes mirrors have the C layout (sizes computed by the host compiler)."""
    src = r'''
#include <stdio.h>
#include "trimmoe.h"
int main(){printf("%zu %zu %zu %zu %zu %zu %zu %zu\n", sizeof(trimmoe_config), sizeof(trimmoe_weights),
 sizeof(trimmoe_tables), sizeof(trimmoe_tokens), sizeof(trimmoe_layer_out), sizeof(trimmoe_stats_t),
 sizeof(trimmoe_feedback_cfg), sizeof(trimmoe_feedback_out));}
'''
    import subprocess
    import tempfile
    with tempfile.TemporaryDirectory() as d:
        p = os.path.join(d, "s.c")
        with open(p, "w") as fh:
            fh.write(src)
        exe = os.path.join(d, "s")
        subprocess.check_call(["gcc", "-I", os.path.join(ROOT, "include"), p, "-o", exe])
        got = [int(x) for x in subprocess.check_output([exe]).split()]
    want = [C.sizeof(x) for x in (B.trimmoe_config, B.trimmoe_weights, B.trimmoe_tables, B.trimmoe_tokens,
                                  B.trimmoe_layer_out, B.trimmoe_stats_t, B.trimmoe_feedback_cfg,
                                  B.trimmoe_feedback_out)]
    assert got == want


def _structs(cfg, **over):
    small = W.make_small_weights(cfg)
    tables = W.make_tables(cfg, small["W_r"])
    tables.update(over)
    c = B.trimmoe_config(N=cfg.N, d=cfg.d, E=cfg.E, k=cfg.k, F=cfg.F, F_sh=cfg.F_sh, C=cfg.C, M=cfg.M,
                         H=cfg.H, act=cfg.act, renorm_topk=0, n_sub=cfg.n_sub, T_max=16, omega_T=0.5,
                         omega_D=0.5, d_ref_ms=float(tables["d_ref"]), phi_beta=0.02, profile=0)
    fake = C.c_void_p(0x1000)           # never dereferenced: validation fails first
    w = B.trimmoe_weights(W_r=fake, b_r=fake, W_x=fake, b_x=fake, W13=fake, W2=fake, W13_sh=None, W2_sh=None)
    keep = {k: np.ascontiguousarray(v) for k, v in tables.items() if k != "d_ref"}
    keep["place"] = keep["place"].astype(np.uint16)
    t = B.trimmoe_tables(place=keep["place"].ctypes.data, sim=keep["sim"].ctypes.data,
                         sub_thresh=keep["sub_thresh"].ctypes.data, trans_ms=keep["trans"].ctypes.data,
                         comp_ms=keep["comp"].ctypes.data, P=keep["P"].ctypes.data,
                         theta=keep["theta"].ctypes.data, lambda_=keep["lam"].ctypes.data,
                         eps=keep["eps"].ctypes.data)
    return c, w, t, keep


def _create(lib, c, w, t):
    h = C.c_void_p()
    rc = lib.trimmoe_create(C.byref(c), C.byref(w), C.byref(t), C.byref(h))
    return rc, h, B.trimmoe_last_error(None)


def test_create_rejects_bad_arguments_on_host(lib):
    cfg = small_cfg()
    c, w, t, keep = _structs(cfg)
    h = C.c_void_p()
    assert lib.trimmoe_create(None, C.byref(w), C.byref(t), C.byref(h)) == -1
    bad = B.trimmoe_config.from_buffer_copy(c)
    bad.d = 200
    rc, _, msg = _create(lib, bad, w, t)
    assert rc == -2 and "256" in msg
    bad = B.trimmoe_config.from_buffer_copy(c)
    bad.k = 9
    assert _create(lib, bad, w, t)[0] == -2
    bad = B.trimmoe_config.from_buffer_copy(c)
    bad.M = 17
    assert _create(lib, bad, w, t)[0] == -2
    bad = B.trimmoe_config.from_buffer_copy(c)
    bad.d_ref_ms = 0.0
    assert _create(lib, bad, w, t)[0] == -1
    bad = B.trimmoe_config.from_buffer_copy(c)
    bad.F_sh = 128                       # shared weights missing
    assert _create(lib, bad, w, t)[0] == -1
    mis = B.trimmoe_weights.from_buffer_copy(w)
    mis.W13 = 0x1003                      # not 16-byte aligned
    assert _create(lib, c, mis, t)[0] == -1
    # attention sublayer of the full block
    bad = B.trimmoe_config.from_buffer_copy(c)
    bad.attn_heads, bad.attn_kv_heads, bad.head_dim, bad.attn_seq, bad.rope_theta = 8, 3, 64, 128, 1e4
    rc, _, msg = _create(lib, bad, w, t)
    assert rc == -1 and "attn_kv_heads" in msg
    bad.attn_kv_heads, bad.head_dim = 2, 96
    rc, _, msg = _create(lib, bad, w, t)
    assert rc == -2 and "head_dim" in msg
    bad.head_dim, bad.attn_seq = 64, 129
    rc, _, msg = _create(lib, bad, w, t)
    assert rc == -2 and "attn_seq" in msg
    bad.attn_seq, bad.attn_heads, bad.attn_kv_heads = 128, 5, 1         # (5 + 2) * 64 = 448
    assert _create(lib, bad, w, t)[0] == -2
    bad.attn_heads, bad.attn_kv_heads = 8, 2
    rc, _, msg = _create(lib, bad, w, t)                                 # weights missing
    assert rc == -1 and "W_qkv" in msg
    place = keep["place"].copy()
    place[2, 5] = 0
    t2 = B.trimmoe_tables.from_buffer_copy(t)
    t2.place = place.ctypes.data
    rc, _, msg = _create(lib, c, w, t2)
    assert rc == -5 and "layer 2" in msg
    P = keep["P"].copy()
    P[0, 0, 0] += 0.5
    t3 = B.trimmoe_tables.from_buffer_copy(t)
    t3.P = P.ctypes.data
    assert _create(lib, c, w, t3)[0] == -1
    tr = keep["trans"].copy()
    tr[0, 1] = -1
    t4 = B.trimmoe_tables.from_buffer_copy(t)
    t4.trans_ms = tr.ctypes.data
    assert _create(lib, c, w, t4)[0] == -1


def test_null_handle_calls_fail_cleanly(lib):
    assert lib.trimmoe_layer_step(None, 0, 1, None, None, None) == -1
    assert lib.trimmoe_watchdog_selftest(None, 1000, None) == -1
    assert lib.trimmoe_forward(None, 1, None, None) == -1
    assert lib.trimmoe_stats(None, None) == -1
    lib.trimmoe_destroy(None)


def _rank_main(rank, world, port, q):
    import bench
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank),
                      MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist = bench.init_dist(world)
    v = bench.max_over_ranks(dist, 10.0 + rank)
    bench.barrier(dist)
    dist.destroy_process_group()
    q.put((rank, v))


def test_replica_timing_reduction_two_ranks():
    """bench.py takes the max step time over ranks (gloo, world size 2)."""
    import multiprocessing as mp
    import socket
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    ps = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in ps:
        p.start()
    for p in ps:
        p.join(timeout=120)
    res = dict(q.get(timeout=5) for _ in range(2))
    assert res == {0: 11.0, 1: 11.0}
