"""Workload recipes: model shapes and restore scenarios, stated as data.

The paper measures Qwen3-0.6B and EXAONE-4.0-1.2B on phones with 8k-32k
contexts (Sec. 6.1); those weights and datasets are not available, so these
synthetic Llama-style shapes with N(0, 0.02) bf16 weights and uniform token
ids stand in for them. RMSNorm eps 1e-5, RoPE theta 500000 (half-split
pairing), no biases, untied LM head, SwiGLU MLP, norm gains 1.
"""
from __future__ import annotations

KV_BF16 = 0
KV_FP16 = 1
KV_F32 = 2  # oracle-only (exact pins); the GPU path stores bf16 or fp16

BLOCK_TOKENS = 16


def shape(n_layers, d_model, n_q_heads, n_kv_heads, head_dim, ffn_dim, vocab,
          kv_dtype=KV_BF16, rope_theta=500000.0, rms_eps=1e-5, max_ctx=None):
    return dict(n_layers=n_layers, d_model=d_model, n_q_heads=n_q_heads,
                n_kv_heads=n_kv_heads, head_dim=head_dim, ffn_dim=ffn_dim,
                vocab=vocab, kv_dtype=kv_dtype, rope_theta=rope_theta,
                rms_eps=rms_eps, block_tokens=BLOCK_TOKENS, max_ctx=max_ctx)


# 2 layers, d 256, 4/2 heads of 64, FFN 688, vocab 1024, bf16 KV.
TINY = shape(2, 256, 4, 2, 64, 688, 1024, KV_BF16, max_ctx=1024)
# 1B-class: 16 layers, d 2048, 32/8 heads of 64, FFN 8192, vocab 128256, fp16 KV.
ONE_B = shape(16, 2048, 32, 8, 64, 8192, 128256, KV_FP16, max_ctx=8192 + 1024)
# 3B-class: 28 layers, d 3072, 24/8 heads of 128, FFN 8192, vocab 128256, bf16 KV.
THREE_B = shape(28, 3072, 24, 8, 128, 8192, 128256, KV_BF16, max_ctx=32768 + 1024)

# Restore scenarios (context tokens, eviction, prompt tokens).
SCENARIOS = {
    # tiny: 512-token context, last 256 tokens evicted backward-out, 32-token prompt
    "tiny": dict(model=TINY, context=512, evict_tail=256, mode="drop", prompt=32),
    # 1B: 8192-token context, 50% tail evicted and restored by recompute, 128-token prompt
    "1b_recompute": dict(model=ONE_B, context=8192, evict_tail=4096, mode="drop", prompt=128),
    # 3B: 32768-token context, 30% of blocks scattered to pinned host, 256-token prompt
    "3b_scattered_copy": dict(model=THREE_B, context=32768, scatter_frac=0.30, prompt=256),
    # 3B mixed: last 8 layers' weights on host, tail >= 16384 dropped,
    # 20% of the remaining blocks copied, 512-token prompt
    "3b_mixed": dict(model=THREE_B, context=32768, weights_evicted=(20, 28),
                     drop_from=16384, scatter_frac=0.20, prompt=512),
    # 3B sweep: evicted fraction of the token tail x {copy, recompute, hybrid}, 128-token prompt
    "3b_sweep": dict(model=THREE_B, context=32768, fractions=(0.0, 0.10, 0.25, 0.50, 0.75, 1.0),
                     policies=("copy", "recompute", "hybrid"), prompt=128),
    # 3B eviction-order ablation (Sec. 6.3): a fraction of the layers (weights and
    # every KV block) swapped to pinned host, chosen backward-out (last layers),
    # forward-out (first layers) or random-out (seeded, several draws); restore
    # forward-in, 128-token prompt
    "3b_order": dict(model=THREE_B, context=32768, fractions=(0.25, 0.50),
                     orders=("backward", "forward", "random"), random_draws=5, prompt=128),
    # swapped token tails of the 3B context restored by copy vs read in place by
    # the attention kernels, 128-token prompt
    "3b_read_swapped": dict(model=THREE_B, context=32768, fractions=(0.10, 0.25, 0.50, 1.0),
                            prompt=128),
    # decode after the first token: single-token steps over a resident context
    "1b_decode": dict(model=ONE_B, context=8192, prompt=1, decode=True),
    "3b_decode": dict(model=THREE_B, context=32768, prompt=1, decode=True),
}


def scaled(model: dict, **over) -> dict:
    """A copy of a model shape with some fields replaced (smaller test cases)."""
    m = dict(model)
    m.update(over)
    return m
