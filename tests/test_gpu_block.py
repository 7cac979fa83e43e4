"""GPU parity of the full block: the attention sublayer (Sec. III-C, attention
placement) in front of every MoE step, through the C ABI, against the oracle.

Per layer the GPU's post-attention state is compared with the oracle's
attention on the live rows, then the oracle's MoE part reads the GPU's
post-attention state and every decision and hidden row is compared as for the
MoE step alone (teacher forcing inside the layer).
"""
import numpy as np
import pytest

from paper_2608_00573_gb300 import binding as B
from paper_2608_00573_gb300 import workload as W
from tests.gpu_helpers import compare_layer, make_engine, targeted_rows
from tests.oracle_helpers import small_cfg

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="session", autouse=True)
def built_library():
    from paper_2608_00573_gb300 import build
    build.build()
    B.lib()


BLOCKS = {
    # grouped-query heads, ragged last sequence, top-2 SwiGLU
    "gqa_h64_s128": small_cfg(name="b1", N=3, d=512, E=8, k=2, F=256, T=700, M=10, H=3, renorm_topk=1,
                              attn_heads=8, attn_kv_heads=2, head_dim=64, attn_seq=128, seed=41),
    # head_dim 128, shared expert, sequence length not a power of two
    "mha_h128_s100_shared": small_cfg(name="b2", N=3, d=512, E=16, k=4, F=128, F_sh=128, T=333, M=10, H=3,
                                      attn_heads=4, attn_kv_heads=4, head_dim=128, attn_seq=100, seed=42),
    # ReLU experts, 64-class exit head, short sequences, exit prediction
    "relu_c64_s37_kc16": small_cfg(name="b3", N=4, d=256, E=8, k=1, F=256, C=64, act=W.ACT_RELU, T=300, M=10,
                                   attn_heads=4, attn_kv_heads=4, head_dim=64, attn_seq=37, n_centroids=16,
                                   seed=43),
    # 4200 tokens: the attention projections and the routed experts (2100 rows
    # per group on average) run on CTA pairs, 256-row tiles with a ragged tail
    "gqa_pair_T4200": small_cfg(name="b5", N=2, d=512, E=4, k=2, F=256, T=4200, M=10, H=3, renorm_topk=1,
                                attn_heads=8, attn_kv_heads=2, head_dim=64, attn_seq=128, seed=44),
    # many (head, sequence) units per attention CTA: 1500 units of three query
    # heads per key/value head, so groups straddle the CTAs' unit ranges and
    # every Q slot and K/V buffer is reused; ragged last sequence
    "gqa3_h64_s8_many_units": small_cfg(name="b6", N=2, d=512, E=8, k=2, F=256, T=1000, M=10, H=3,
                                        renorm_topk=1, attn_heads=12, attn_kv_heads=4, head_dim=64, attn_seq=8,
                                        seed=45),
    # the same at head_dim 128: 978 units, ragged last sequence of 4 tokens
    "gqa3_h128_s8_many_units": small_cfg(name="b7", N=2, d=512, E=8, k=2, F=256, T=1300, M=10, H=3,
                                         renorm_topk=1, attn_heads=6, attn_kv_heads=2, head_dim=128, attn_seq=8,
                                         seed=46),
}


# exit-head bias per configuration: the 64-class head's max-softmax confidence
# needs a larger bias than the sigmoid head to reach p_J = 0.9
EXIT_BIAS = {"gqa_h64_s128": 1.0, "mha_h128_s100_shared": 1.0, "relu_c64_s37_kc16": 5.0, "gqa_pair_T4200": 1.0,
             "gqa3_h64_s8_many_units": 1.0, "gqa3_h128_s8_many_units": 1.0}


@pytest.mark.parametrize("name", list(BLOCKS))
def test_full_block_parity_small(name):
    import torch
    cfg = BLOCKS[name]
    eng, om, tables, small, experts = make_engine(cfg, theta=0.9, exit_bias=EXIT_BIAS[name])
    dev = eng.tokens_to_device(W.make_tokens(cfg))
    reports = [compare_layer(cfg, om, eng, l, dev, experts) for l in range(cfg.N)]
    tot = {k: sum(r[k] for r in reports) for k in ("exec", "skip", "exit", "near_mismatch")}
    print(name, tot, [round(r["attn_rel_err"], 5) for r in reports], [round(r["max_rel_err"], 5) for r in reports])
    assert tot["exec"] > 0 and tot["skip"] > 0 and tot["exit"] > 0, tot
    eng.close()
    torch.cuda.synchronize()


def test_full_block_single_token_sequences_and_tiny_batches():
    """attn_seq = 1 (every token attends to itself only), T = 1 and T = 5."""
    import torch
    cfg = small_cfg(name="b4", N=2, d=256, E=8, k=2, F=256, T=5, M=10, attn_heads=4, attn_kv_heads=2,
                    head_dim=64, attn_seq=1, seed=44)
    for T in (1, 5):
        eng, om, tables, small, experts = make_engine(cfg.replace(T=T), theta=0.9, exit_bias=1.0)
        dev = eng.tokens_to_device(W.make_tokens(cfg, T=T))
        for l in range(cfg.N):
            compare_layer(cfg, om, eng, l, dev, experts)
        eng.close()
    torch.cuda.synchronize()


def test_full_block_mixtral_shape_sampled():
    """Mixtral-shaped full block (32 query / 8 key-value heads of 128, d = 4096,
    user sequences of 128) over 4200 tokens, so that the attention projections
    run on CTA pairs with a ragged last tile and the last sequence is ragged.
    Every decision is compared; the attention output and the hidden state on
    rows aimed at the tile structure: the first and last token of every
    128-token block (every row tile of the q/k/v and output projections, both
    CTAs of each pair tile, and the first and last position of every
    sequence), plus the MoE GEMMs' group edges and every 128-row block of every
    expert group in the compacted order."""
    import torch
    base = W.with_attention(W.CONFIGS["mixtral"])
    T = 4200
    cfg = base.replace(N=2, T=T)
    eng, om, tables, small, experts = make_engine(cfg, device_experts=True)
    dev = eng.tokens_to_device(W.make_tokens(cfg))
    edges = np.unique(np.concatenate([np.arange(0, T, 128), np.minimum(np.arange(127, T + 127, 128), T - 1)]))

    def rows(g):
        return np.union1d(edges, targeted_rows(g, T, cfg.k, cfg.E, tiles=True, extra=16, seed=5))

    for l in range(cfg.N):
        r = compare_layer(cfg, om, eng, l, dev, experts, row_sample=rows)
        print(l, r["exec"], r["skip"], r["exit"], r["attn_rel_err"], r["max_rel_err"], r["rows_checked"])
    eng.close()
    torch.cuda.synchronize()
