"""Pins for the fp64 oracle (CPU only).

The oracle is only trusted after it agrees with things that are fixed
independently of it:
  * brute-force dense attention on the logical (un-paged) arrays, which never
    touches a block table;
  * closed forms: a single cached token returns exactly that token's value
    row; constant V returns V; a zero query, a zero scale or identical keys
    return the plain mean of V;
  * invariance of the result to relabelling physical block ids;
  * invariance to cutting the context into chunks merged by log-sum-exp;
  * grouped-query attention equals multi-head attention over KV heads that
    are repeated g times;
  * torch's fp64 scaled_dot_product_attention on tiny dense shapes.
A last group plants mistakes in a copy of the oracle source and checks that
the pins catch every one of them.
"""
import math
import os
import re
import shutil
import subprocess
import tempfile

import numpy as np
import pytest
import torch

import oracle
from paper_2608_21719_gb300 import inputs


def _logical_case(S, Hq, Hkv, d, bs, lengths, seed, spare=3):
    gen = torch.Generator().manual_seed(seed)
    q = torch.randn((S, Hq, d), generator=gen).to(torch.bfloat16)
    kl = [torch.randn((int(L), Hkv, d), generator=gen).to(torch.bfloat16) for L in lengths]
    vl = [torch.randn((int(L), Hkv, d), generator=gen).to(torch.bfloat16) for L in lengths]
    mbps = max(1, max((int(L) + bs - 1) // bs for L in lengths) + 1)
    nb = inputs.blocks_needed(np.asarray(lengths), bs) + spare
    bt = inputs.build_block_table(np.asarray(lengths, dtype=np.int32), bs, mbps, nb,
                                  np.random.default_rng(seed + 7))
    k, v = inputs.scatter_logical(kl, vl, Hkv, bs, bt, nb)
    return q, kl, vl, k, v, bt, np.asarray(lengths, dtype=np.int32)


def _run(lib, q, k, v, bt, lens, Hkv, scale, chunk=0, threads=4):
    return oracle.decode_attention(inputs.bf16_bits(q), inputs.bf16_bits(k), inputs.bf16_bits(v),
                                   bt, lens, Hkv, scale, chunk_tokens=chunk, num_threads=threads,
                                   lib=lib)


def _dense(q, kl, vl, Hkv, scale):
    """Attention straight from the definition on logical arrays (float64)."""
    S, Hq, d = q.shape
    g = Hq // Hkv
    out = np.zeros((S, Hq, d))
    qd = q.double().numpy()
    for s in range(S):
        L = kl[s].shape[0]
        if L == 0:
            continue
        K = kl[s].double().numpy()
        V = vl[s].double().numpy()
        for h in range(Hq):
            x = scale * (K[:, h // g, :] @ qd[s, h])
            w = np.exp(x - x.max())
            out[s, h] = (w[:, None] * V[:, h // g, :]).sum(0) / w.sum()
    return out


SHAPES = [
    # S, Hq, Hkv, d, bs, lengths
    (3, 8, 2, 128, 16, [1, 37, 64]),
    (4, 4, 4, 32, 8, [5, 8, 9, 23]),
    (2, 5, 1, 16, 4, [13, 4]),
    (3, 8, 8, 8, 16, [16, 17, 15]),
]


def _battery(lib):
    """Every pin, run against ``lib``; returns the names of those that fail."""
    failed = []
    for i, (S, Hq, Hkv, d, bs, lens) in enumerate(SHAPES):
        q, kl, vl, k, v, bt, L = _logical_case(S, Hq, Hkv, d, bs, lens, seed=100 + i)
        scale = 1.0 / math.sqrt(d)
        try:
            got = _run(lib, q, k, v, bt, L, Hkv, scale)
        except RuntimeError:
            failed.append("run%d" % i)
            continue
        ref = _dense(q, kl, vl, Hkv, scale)
        if not np.allclose(got, ref, rtol=1e-12, atol=1e-12):
            failed.append("brute_force%d" % i)
        # GQA == MHA with each KV head repeated g times.
        g = Hq // Hkv
        k_rep = k.repeat_interleave(g, dim=1)
        v_rep = v.repeat_interleave(g, dim=1)
        try:
            got_mha = _run(lib, q, k_rep, v_rep, bt, L, Hq, scale)
            if not np.array_equal(got, got_mha):
                failed.append("gqa_mha%d" % i)
        except RuntimeError:
            failed.append("gqa_mha%d" % i)
    # Closed forms on one shape.
    S, Hq, Hkv, d, bs = 2, 4, 2, 64, 16
    q, kl, vl, k, v, bt, L = _logical_case(S, Hq, Hkv, d, bs, [1, 40], seed=7)
    scale = 1.0 / math.sqrt(d)
    try:
        out = _run(lib, q, k, v, bt, L, Hkv, scale)
        g = Hq // Hkv
        for h in range(Hq):  # a single cached token returns its value row exactly
            if not np.array_equal(out[0, h], vl[0][0, h // g].double().numpy()):
                failed.append("single_token")
                break
        vc = [torch.ones_like(x) * 0.375 for x in vl]  # constant V returns V
        kk, vv = inputs.scatter_logical(kl, vc, Hkv, bs, bt, k.shape[0])
        oc = _run(lib, q, kk, vv, bt, L, Hkv, scale)
        if not np.allclose(oc, 0.375, rtol=0, atol=1e-14):
            failed.append("constant_v")
        # zero query / zero scale / identical keys all give the mean of V
        mean = np.stack([[vl[s][:, h // g].double().numpy().mean(0) for h in range(Hq)] for s in range(S)])
        oz = _run(lib, torch.zeros_like(q), k, v, bt, L, Hkv, scale)
        if not np.allclose(oz, mean, rtol=0, atol=1e-13):
            failed.append("zero_query")
        os_ = _run(lib, q, k, v, bt, L, Hkv, 0.0)
        if not np.allclose(os_, mean, rtol=0, atol=1e-13):
            failed.append("zero_scale")
        ke = [x[:1].expand_as(x).contiguous() for x in kl]
        kk, vv = inputs.scatter_logical(ke, vl, Hkv, bs, bt, k.shape[0])
        oe = _run(lib, q, kk, vv, bt, L, Hkv, scale)
        if not np.allclose(oe, mean, rtol=0, atol=1e-13):
            failed.append("equal_keys")
    except RuntimeError:
        failed.append("closed_forms_run")
    return failed


def test_oracle_passes_every_pin():
    assert _battery(oracle.load()) == []


@pytest.mark.parametrize("S,Hq,Hkv,d,bs,lens", SHAPES)
def test_brute_force_dense(S, Hq, Hkv, d, bs, lens):
    q, kl, vl, k, v, bt, L = _logical_case(S, Hq, Hkv, d, bs, lens, seed=11)
    scale = 1.0 / math.sqrt(d)
    got = _run(oracle.load(), q, k, v, bt, L, Hkv, scale)
    np.testing.assert_allclose(got, _dense(q, kl, vl, Hkv, scale), rtol=1e-12, atol=1e-12)


def test_single_token_returns_value_row_exactly():
    q, kl, vl, k, v, bt, L = _logical_case(3, 8, 2, 128, 16, [1, 1, 1], seed=5)
    out = _run(oracle.load(), q, k, v, bt, L, 2, 1.0 / math.sqrt(128))
    for s in range(3):
        for h in range(8):
            assert np.array_equal(out[s, h], vl[s][0, h // 4].double().numpy())


def test_empty_sequence_gives_zeros():
    q, kl, vl, k, v, bt, L = _logical_case(3, 4, 2, 16, 4, [0, 5, 0], seed=6)
    out = _run(oracle.load(), q, k, v, bt, L, 2, 0.25)
    assert np.all(out[0] == 0) and np.all(out[2] == 0)
    assert np.all(np.isfinite(out[1]))


def test_block_relabelling_invariance_bit_exact():
    S, Hq, Hkv, d, bs = 4, 8, 2, 128, 16
    lens = [37, 200, 16, 95]
    q, kl, vl, k, v, bt, L = _logical_case(S, Hq, Hkv, d, bs, lens, seed=21)
    out_a = _run(oracle.load(), q, k, v, bt, L, Hkv, 0.1)
    nb = k.shape[0]
    bt2 = inputs.build_block_table(L, bs, bt.shape[1], nb, np.random.default_rng(999))
    assert not np.array_equal(bt, bt2)
    k2, v2 = inputs.scatter_logical(kl, vl, Hkv, bs, bt2, nb)
    out_b = _run(oracle.load(), q, k2, v2, bt2, L, Hkv, 0.1)
    assert np.array_equal(out_a, out_b)


@pytest.mark.parametrize("chunk", [1, 7, 16, 64, 256, 1 << 20])
def test_chunked_lse_merge_matches_definition(chunk):
    S, Hq, Hkv, d, bs = 3, 8, 2, 128, 16
    q, kl, vl, k, v, bt, L = _logical_case(S, Hq, Hkv, d, bs, [1, 300, 517], seed=31)
    scale = 1.0 / math.sqrt(d)
    full = _run(oracle.load(), q, k, v, bt, L, Hkv, scale)
    split = _run(oracle.load(), q, k, v, bt, L, Hkv, scale, chunk=chunk)
    np.testing.assert_allclose(split, full, rtol=0, atol=1e-12)


def test_torch_sdpa_fp64_cross_check():
    S, Hq, Hkv, d, bs = 2, 8, 2, 64, 8
    q, kl, vl, k, v, bt, L = _logical_case(S, Hq, Hkv, d, bs, [33, 12], seed=41)
    scale = 1.0 / math.sqrt(d)
    got = _run(oracle.load(), q, k, v, bt, L, Hkv, scale)
    g = Hq // Hkv
    for s in range(S):
        qs = q[s].double()[None, :, None, :]                       # [1, Hq, 1, d]
        ks = kl[s].double().permute(1, 0, 2).repeat_interleave(g, 0)[None]  # [1, Hq, L, d]
        vs = vl[s].double().permute(1, 0, 2).repeat_interleave(g, 0)[None]
        ref = torch.nn.functional.scaled_dot_product_attention(qs, ks, vs, scale=scale)
        np.testing.assert_allclose(got[s], ref[0, :, 0, :].numpy(), rtol=1e-12, atol=1e-12)


def test_bad_block_id_and_overlong_sequence_are_errors():
    q, kl, vl, k, v, bt, L = _logical_case(2, 4, 2, 16, 4, [5, 9], seed=51)
    bad = bt.copy()
    bad[1, 1] = k.shape[0]
    with pytest.raises(RuntimeError, match="block id"):
        _run(oracle.load(), q, k, v, bad, L, 2, 0.25)
    too_long = L.copy()
    too_long[0] = bt.shape[1] * 4 + 1
    with pytest.raises(RuntimeError, match="longer"):
        _run(oracle.load(), q, k, v, bt, too_long, 2, 0.25)


def test_kv_byte_accounting_matches_paper_figure():
    from paper_2608_21719_gb300 import roofline
    golden = {}
    with open(os.path.join(os.path.dirname(__file__), "golden", "kv_bytes_llama70b.txt")) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                key, val = line.split()
                golden[key] = float(val)
    per_layer = roofline.kv_bytes_per_token(int(golden["num_kv_heads"]), int(golden["head_dim"]),
                                            int(golden["elem_bytes"]))
    assert per_layer == 4096
    per_token = per_layer * int(golden["layers"])
    assert per_token == golden["kib_per_token"] * 1024
    chain = per_token * int(golden["chain_tokens"])
    assert round(chain / 1e9, 1) == golden["chain_gb_1dp"]
    b = roofline.algorithmic_bytes([4096], 64, 8, 128, 16)
    assert b["kv"] == 4096 * 4096


# --- planted mistakes: each must be caught by the battery ------------------

MUTATIONS = {
    "kv_head_mapping_modulo": (r"const int j = h / g;", "const int j = h % jb->num_kv_heads;"),
    "scale_dropped": (r"logits\[t\] = jb->scale \* dot;", "logits[t] = dot;"),
    "layout_slot_major": (
        r"return cache \+ \(page \* jb->block_size \+ \(size_t\)\(t % jb->block_size\)\) \* jb->head_dim;",
        "return cache + (((size_t)b * jb->block_size + (size_t)(t % jb->block_size)) * jb->num_kv_heads"
        " + (size_t)j) * jb->head_dim;"),
    "no_normalisation": (r"for \(int i = 0; i < d; \+\+i\) o\[i\] /= z;", "for (int i = 0; i < d; ++i) o[i] /= 1.0;"),
    "first_token_dropped": (r"for \(int t = 0; t < L; \+\+t\) \{\n        double w", "for (int t = 1; t < L; ++t) {\n        double w"),
    "query_of_kv_head": (r"jb->q \+ \(\(size_t\)s \* jb->num_q_heads \+ h\) \* d;",
                         "jb->q + ((size_t)s * jb->num_q_heads + j) * d;"),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_mistake_is_caught(name, tmp_path):
    if shutil.which("gcc") is None:
        pytest.skip("gcc not available")
    pattern, repl = MUTATIONS[name]
    src = open(os.path.join(os.path.dirname(oracle.__file__), "ps_oracle.c")).read()
    mutated, n = re.subn(pattern, lambda m: repl, src)
    assert n >= 1, "mutation %s no longer applies to the oracle source" % name
    path = tmp_path / "mut.c"
    path.write_text(mutated)
    so = str(tmp_path / ("libmut_%s.so" % name))
    oracle.build(force=True, src=str(path), out=so)
    failed = _battery(oracle.load(so))
    assert failed, "planted mistake %s passed every pin" % name


# --- KV hand-off pack / unpack -------------------------------------------

def _handoff_case(seed, Hkv=2, d=16, bs=8, lens=(5, 0, 17, 8)):
    gen = torch.Generator().manual_seed(seed)
    kl = [torch.randn((L, Hkv, d), generator=gen).to(torch.bfloat16) for L in lens]
    vl = [torch.randn((L, Hkv, d), generator=gen).to(torch.bfloat16) for L in lens]
    L = np.asarray(lens, dtype=np.int32)
    nb = inputs.blocks_needed(L, bs) + 3
    bt = inputs.build_block_table(L, bs, max(1, int(L.max()) // bs + 2), nb, np.random.default_rng(seed))
    k, v = inputs.scatter_logical(kl, vl, Hkv, bs, bt, nb)
    return kl, vl, k, v, bt, L


def test_pack_equals_logical_arrays():
    kl, vl, k, v, bt, L = _handoff_case(61)
    packed = oracle.kv_pack(inputs.bf16_bits(k), inputs.bf16_bits(v), bt, L)
    off = oracle.packed_offsets(L, 2, 16)
    for i, n in enumerate(L):
        kp = packed[off[i]:off[i] + 2 * n * 16].reshape(2, n, 16)
        vp = packed[off[i] + 2 * n * 16:off[i] + 4 * n * 16].reshape(2, n, 16)
        assert np.array_equal(kp, inputs.bf16_bits(kl[i].permute(1, 0, 2)))
        assert np.array_equal(vp, inputs.bf16_bits(vl[i].permute(1, 0, 2)))


def test_unpack_into_another_pool_then_pack_round_trips():
    kl, vl, k, v, bt, L = _handoff_case(62)
    packed = oracle.kv_pack(inputs.bf16_bits(k), inputs.bf16_bits(v), bt, L)
    # receiver: a different pool size and a different permutation
    nb2 = inputs.blocks_needed(L, 8) + 9
    bt2 = inputs.build_block_table(L, 8, bt.shape[1], nb2, np.random.default_rng(7))
    k2 = np.full((nb2, 2, 8, 16), 0x7fc0, dtype=np.uint16)  # NaN everywhere
    v2 = k2.copy()
    k2u, v2u = oracle.kv_unpack(packed, k2, v2, bt2, L)
    again = oracle.kv_pack(k2u, v2u, bt2, L)
    assert np.array_equal(again, packed)
    # slots that no sequence owns keep their old bits
    owned = np.zeros(k2.shape[:1] + k2.shape[2:3], dtype=bool)
    for i, n in enumerate(L):
        for t in range(int(n)):
            owned[bt2[i, t // 8], t % 8] = True
    for b in range(nb2):
        for t in range(8):
            if not owned[b, t]:
                assert np.all(k2u[b, :, t] == 0x7fc0) and np.all(v2u[b, :, t] == 0x7fc0)


def test_pack_is_invariant_to_block_relabelling():
    kl, vl, k, v, bt, L = _handoff_case(63)
    a = oracle.kv_pack(inputs.bf16_bits(k), inputs.bf16_bits(v), bt, L)
    nb = k.shape[0]
    bt2 = inputs.build_block_table(L, 8, bt.shape[1], nb, np.random.default_rng(99))
    k2, v2 = inputs.scatter_logical(kl, vl, 2, 8, bt2, nb)
    b = oracle.kv_pack(inputs.bf16_bits(k2), inputs.bf16_bits(v2), bt2, L)
    assert np.array_equal(a, b)


def test_pack_rejects_block_outside_pool():
    kl, vl, k, v, bt, L = _handoff_case(64)
    bad = bt.copy()
    bad[2, 1] = k.shape[0] + 3
    with pytest.raises(RuntimeError, match="block id"):
        oracle.kv_pack(inputs.bf16_bits(k), inputs.bf16_bits(v), bad, L)


# --- chunked prefill -----------------------------------------------------

def _prefill_case(seed, Hq=8, Hkv=2, d=32, bs=8, lens=(20, 9, 33), qlens=(7, 9, 1)):
    gen = torch.Generator().manual_seed(seed)
    kl = [torch.randn((L, Hkv, d), generator=gen).to(torch.bfloat16) for L in lens]
    vl = [torch.randn((L, Hkv, d), generator=gen).to(torch.bfloat16) for L in lens]
    T = int(sum(qlens))
    q = torch.randn((T, Hq, d), generator=gen).to(torch.bfloat16)
    L = np.asarray(lens, dtype=np.int32)
    qs = np.concatenate([[0], np.cumsum(qlens)]).astype(np.int32)
    nb = inputs.blocks_needed(L, bs) + 2
    bt = inputs.build_block_table(L, bs, int(L.max()) // bs + 2, nb, np.random.default_rng(seed))
    k, v = inputs.scatter_logical(kl, vl, Hkv, bs, bt, nb)
    return q, kl, vl, k, v, bt, L, qs


def _prefill_dense(q, kl, vl, L, qs, Hkv, scale):
    T, Hq, d = q.shape
    g = Hq // Hkv
    out = np.zeros((T, Hq, d))
    for s in range(len(L)):
        K = kl[s].double().numpy()
        V = vl[s].double().numpy()
        Q = int(qs[s + 1] - qs[s])
        for i in range(Q):
            p = int(L[s]) - Q + i
            for h in range(Hq):
                x = scale * (K[:p + 1, h // g] @ q[qs[s] + i, h].double().numpy())
                w = np.exp(x - x.max())
                out[qs[s] + i, h] = (w[:, None] * V[:p + 1, h // g]).sum(0) / w.sum()
    return out


def test_prefill_matches_causal_brute_force():
    q, kl, vl, k, v, bt, L, qs = _prefill_case(71)
    got = oracle.prefill_attention(inputs.bf16_bits(q), inputs.bf16_bits(k), inputs.bf16_bits(v), bt, L, qs, 2, 0.2)
    np.testing.assert_allclose(got, _prefill_dense(q, kl, vl, L, qs, 2, 0.2), rtol=1e-12, atol=1e-12)


def test_prefill_with_one_query_per_sequence_is_decode_bit_exact():
    q, kl, vl, k, v, bt, L, qs = _prefill_case(72, qlens=(1, 1, 1))
    pre = oracle.prefill_attention(inputs.bf16_bits(q), inputs.bf16_bits(k), inputs.bf16_bits(v), bt, L, qs, 2, 0.3)
    dec = oracle.decode_attention(inputs.bf16_bits(q), inputs.bf16_bits(k), inputs.bf16_bits(v), bt, L, 2, 0.3)
    assert np.array_equal(pre, dec)


def test_prefill_full_prompt_matches_torch_causal_sdpa():
    lens = (24, 16)
    q, kl, vl, k, v, bt, L, qs = _prefill_case(73, lens=lens, qlens=lens)
    got = oracle.prefill_attention(inputs.bf16_bits(q), inputs.bf16_bits(k), inputs.bf16_bits(v), bt, L, qs, 2, 0.25)
    for s in range(2):
        Qs = q[qs[s]:qs[s + 1]].double().permute(1, 0, 2)[None]                 # [1, Hq, L, d]
        Ks = kl[s].double().permute(1, 0, 2).repeat_interleave(4, 0)[None]
        Vs = vl[s].double().permute(1, 0, 2).repeat_interleave(4, 0)[None]
        ref = torch.nn.functional.scaled_dot_product_attention(Qs, Ks, Vs, is_causal=True, scale=0.25)
        np.testing.assert_allclose(got[qs[s]:qs[s + 1]], ref[0].permute(1, 0, 2).numpy(), rtol=1e-12, atol=1e-12)


def test_prefill_ignores_tokens_after_each_query():
    q, kl, vl, k, v, bt, L, qs = _prefill_case(74, lens=(30,), qlens=(10,))
    a = oracle.prefill_attention(inputs.bf16_bits(q), inputs.bf16_bits(k), inputs.bf16_bits(v), bt, L, qs, 2, 0.2)
    # change K/V of the last 4 tokens: queries at positions < 26 must not move
    kl2 = [kl[0].clone()]
    vl2 = [vl[0].clone()]
    kl2[0][26:] = 7.0
    vl2[0][26:] = -5.0
    k2, v2 = inputs.scatter_logical(kl2, vl2, 2, 8, bt, k.shape[0])
    b = oracle.prefill_attention(inputs.bf16_bits(q), inputs.bf16_bits(k2), inputs.bf16_bits(v2), bt, L, qs, 2, 0.2)
    assert np.array_equal(a[:6], b[:6])          # positions 20..25
    assert not np.allclose(a[6:], b[6:])         # positions 26..29 see the change


def test_planted_prefill_off_by_one_is_caught(tmp_path):
    if shutil.which("gcc") is None:
        pytest.skip("gcc not available")
    src = open(os.path.join(os.path.dirname(oracle.__file__), "ps_oracle.c")).read()
    mutated, n = re.subn(r"for \(int t = 0; t <= p; \+\+t\)", "for (int t = 0; t < p; ++t)", src)
    assert n == 2
    path = tmp_path / "mut.c"
    path.write_text(mutated)
    so = str(tmp_path / "libmut_prefill.so")
    oracle.build(force=True, src=str(path), out=so)
    q, kl, vl, k, v, bt, L, qs = _prefill_case(75)
    try:
        got = oracle.prefill_attention(inputs.bf16_bits(q), inputs.bf16_bits(k), inputs.bf16_bits(v), bt, L, qs, 2,
                                       0.2, lib=oracle.load(so))
        caught = not np.allclose(got, _prefill_dense(q, kl, vl, L, qs, 2, 0.2), rtol=1e-12, atol=1e-12)
    except RuntimeError:
        caught = True
    assert caught
