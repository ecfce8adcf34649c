"""Algorithmic byte accounting for paged decode attention.

The minimum traffic one call must move: every cached K and V element of
every sequence once, the queries, the outputs, the block-table entries that
are read and the sequence lengths.  Split-KV workspace traffic is overhead,
not algorithmic, and is deliberately left out.

Grounding: PowerSlider App. B.2, Eq. (bytes-layer) charges a decode layer
``2 B S d b_w`` bytes of KV cache (K and V, B sequences of context S); with
grouped-query heads the KV width is ``num_kv_heads * head_dim`` rather than
the model width ``d``.  Sec. 3 Obs. 3 quotes 320 KiB of KV per token for
Llama-70B (80 layers, 8 KV heads, head_dim 128, bf16), i.e. 4096 B per token
per layer, which pins ``kv_bytes_per_token``.
"""
from __future__ import annotations

import numpy as np


def kv_bytes_per_token(num_kv_heads: int, head_dim: int, elem_bytes: int = 2) -> int:
    """K and V bytes that one cached token holds in one layer."""
    return 2 * num_kv_heads * head_dim * elem_bytes


def algorithmic_bytes(seq_lens, num_q_heads: int, num_kv_heads: int, head_dim: int,
                      block_size: int, elem_bytes: int = 2) -> dict:
    L = np.asarray(seq_lens, dtype=np.int64)
    S = int(L.shape[0])
    kv = int(L.sum()) * kv_bytes_per_token(num_kv_heads, head_dim, elem_bytes)
    q = S * num_q_heads * head_dim * elem_bytes
    out = S * num_q_heads * head_dim * elem_bytes
    bt = int(((L + block_size - 1) // block_size).sum()) * 4
    sl = S * 4
    return {"kv": kv, "q": q, "out": out, "block_table": bt, "seq_lens": sl,
            "total": kv + q + out + bt + sl}


def decode_flops(seq_lens, num_q_heads: int, head_dim: int) -> int:
    """Q.K^T and P.V multiply-adds, 2 flops each: 4 * sum(L) * Hq * d
    (the attention term 4BSd of Eq. (flops-layer), per query head)."""
    return 4 * int(np.asarray(seq_lens, dtype=np.int64).sum()) * num_q_heads * head_dim


def prefill_flops(seq_lens, q_lens, num_q_heads: int, head_dim: int) -> int:
    """Causal chunked prefill: query i of a sequence with L cached tokens,
    the last Q of them new, sees L - Q + i + 1 keys; each key costs a
    Q.K^T and a P.V multiply-add per head dimension (4 flops).  Summed over
    a sequence: Q (L - Q) + Q (Q + 1) / 2 query-key pairs per query head."""
    L = np.asarray(seq_lens, dtype=np.int64)
    Q = np.asarray(q_lens, dtype=np.int64)
    pairs = Q * (L - Q) + Q * (Q + 1) // 2
    return 4 * int(pairs.sum()) * num_q_heads * head_dim


def prefill_bytes(seq_lens, q_lens, num_q_heads: int, num_kv_heads: int, head_dim: int,
                  elem_bytes: int = 2) -> int:
    """Compulsory HBM bytes of one prefill call: each sequence's K/V once,
    the queries and the outputs."""
    L = np.asarray(seq_lens, dtype=np.int64)
    T = int(np.asarray(q_lens, dtype=np.int64).sum())
    return int(L.sum()) * kv_bytes_per_token(num_kv_heads, head_dim, elem_bytes) + \
        2 * T * num_q_heads * head_dim * elem_bytes
