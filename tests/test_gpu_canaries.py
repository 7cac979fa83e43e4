"""Guard bands around every caller-owned array the library writes.

Each token-state array, the hidden rows and every layer output are copied into
the middle of a byte buffer whose leading and trailing 512 bytes hold a canary
pattern; layer steps and a forward at ragged token counts (not multiples of
32, 128 or 256) must leave the bands untouched: no kernel writes past the T
rows it was given."""
import pytest

from paper_2608_00573_gb300 import binding as B
from paper_2608_00573_gb300 import workload as W
from tests.gpu_helpers import make_engine
from tests.oracle_helpers import small_cfg

pytestmark = pytest.mark.gpu

CANARY = 0xA5
PAD = 512          # bytes; keeps the arrays' 256-byte alignment


@pytest.fixture(scope="session", autouse=True)
def built_library():
    from paper_2608_00573_gb300 import build
    build.build()
    B.lib()


def _guarded(t):
    import torch
    flat = t.contiguous().reshape(-1).view(torch.uint8)
    raw = torch.full((PAD + flat.numel() + PAD,), CANARY, dtype=torch.uint8, device=t.device)
    raw[PAD:PAD + flat.numel()].copy_(flat)
    view = raw[PAD:PAD + flat.numel()].view(t.dtype).reshape(t.shape)
    return view, raw


def _intact(raw):
    return bool((raw[:PAD] == CANARY).all()) and bool((raw[-PAD:] == CANARY).all())


CONFIGS = {
    # routed + shared expert, top-4 of 16
    "moe_shared": small_cfg(name="c1", N=3, d=512, E=16, k=4, F=384, F_sh=256, T=1000, M=10, H=3,
                            zipf_s=0.8, seed=61),
    # full block: attention sublayer (writes the post-attention rows too)
    "block_gqa": small_cfg(name="c2", N=2, d=512, E=8, k=2, F=256, T=1000, M=10, H=3, attn_heads=8,
                           attn_kv_heads=2, head_dim=64, attn_seq=128, seed=62),
}


@pytest.mark.parametrize("name,T", [("moe_shared", 777), ("moe_shared", 1), ("block_gqa", 333)])
def test_outputs_keep_their_guard_bands(name, T):
    import torch
    cfg = CONFIGS[name]
    eng, om, tables, small, experts = make_engine(cfg, T_max=cfg.T, theta=0.9, exit_bias=1.0)
    base = eng.tokens_to_device(W.make_tokens(cfg, T=T))
    g_tok = {k: _guarded(v) for k, v in base.items()}
    tok = {k: v for k, (v, _) in g_tok.items()}
    g_out = {k: (_guarded(v) if v is not None else None) for k, v in eng.alloc_layer_out(T).items()}
    out = {k: (g[0] if g is not None else None) for k, g in g_out.items()}
    for l in range(cfg.N):
        eng.layer_step(l, tok, T=T, out=out)
    g_fwd = {k: _guarded(v) for k, v in base.items()}
    eng.forward({k: v for k, (v, _) in g_fwd.items()}, T=T)
    torch.cuda.synchronize()
    bands = [("step " + k, raw) for k, (_, raw) in g_tok.items()]
    bands += [("out " + k, g[1]) for k, g in g_out.items() if g is not None]
    bands += [("forward " + k, raw) for k, (_, raw) in g_fwd.items()]
    broken = [n for n, raw in bands if not _intact(raw)]
    assert not broken, broken
    eng.close()
