"""GPU parity of the tcgen05 chunked-prefill path against the fp64 oracle.

Tolerance as for decode: max |gpu - oracle| <= 8e-3 (plus the bf16 output
rounding 2^-8 |ref| on custom edge cases, whose short contexts give large
outputs) and mean <= 1e-3, every output finite.  The full-size workload is
compared on every output.  Sampled rows of the 8192-token chunk are also
checked against the decode oracle: causal prefill row i of a sequence is
decode attention over the first p + 1 = L - Q + i + 1 tokens.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_21719_gb300 import inputs

pytestmark = pytest.mark.gpu

MAX_ABS = 8e-3
MEAN_ABS = 1e-3
BF16_REL = 2.0 ** -8


@pytest.fixture(scope="module")
def psd():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_21719_gb300 import build
    build.build()
    from paper_2608_21719_gb300 import ps_decode
    return ps_decode


def _oracle(wl):
    return oracle.prefill_attention(inputs.bf16_bits(wl.q), inputs.bf16_bits(wl.k_cache),
                                    inputs.bf16_bits(wl.v_cache), wl.block_table.cpu().numpy(), wl.lengths,
                                    wl.q_start.cpu().numpy(), wl.k_cache.shape[1], wl.scale)


def _gpu(psd, wl, out=None):
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = psd.prefill_attention(wl.q, wl.k_cache, wl.v_cache, wl.block_table, wl.seq_lens, wl.q_start,
                                wl.max_q_len, out=out, scale=wl.scale, device_status=status)
    torch.cuda.synchronize()
    return out, int(status.item())


def _compare(got, ref, what="", rel=BF16_REL):
    got = got.float().cpu().numpy().astype(np.float64)
    assert np.all(np.isfinite(got)), "non-finite output %s" % what
    err = np.abs(got - ref)
    excess = err - (MAX_ABS + rel * np.abs(ref))
    assert excess.max() <= 0, "%s max abs err %.3g (at |ref| %.3g)" % (
        what, err.max(), np.abs(ref).flat[int(np.argmax(excess))])
    assert err.mean() <= MEAN_ABS, "%s mean abs err %.3g" % (what, err.mean())


def test_tiny_prefill_full_parity(psd):
    wl = inputs.make_prefill_workload("p1", device="cpu", spare_blocks=4).to("cuda")
    out, status = _gpu(psd, wl)
    assert status == 0
    _compare(out, _oracle(wl), "p1", rel=0.0)


# (new tokens, prior tokens) per sequence: one-token chunks, whole prompts,
# chunks that end exactly on / just past a 128-key tile, ragged query tiles,
# and an empty chunk.
EDGE_NEW = [1, 1, 31, 32, 33, 128, 129, 300, 0, 77, 256]
EDGE_PRIOR = [0, 200, 0, 96, 95, 0, 127, 1, 50, 1000, 384]


@pytest.mark.parametrize("Hq,Hkv", [(8, 8), (4, 2), (8, 2), (32, 8), (64, 8), (12, 2), (16, 1)])
@pytest.mark.parametrize("bs", [16, 32, 48])
def test_prefill_edge_chunks_groups_and_block_sizes(psd, Hq, Hkv, bs):
    wl = inputs.make_prefill_workload("p1", device="cpu", new=EDGE_NEW, prior=EDGE_PRIOR, num_q_heads=Hq,
                                      num_kv_heads=Hkv, block_size=bs, spare_blocks=3,
                                      seed=Hq * 31 + bs).to("cuda")
    out, status = _gpu(psd, wl)
    assert status == 0
    _compare(out, _oracle(wl), "edge Hq=%d Hkv=%d bs=%d" % (Hq, Hkv, bs))


def test_prefill_one_token_chunks_match_decode_path(psd):
    """Q_s = 1 everywhere is a decode step; both kernels must agree with the
    same oracle on the same inputs."""
    lens = np.asarray([1, 17, 128, 129, 700, 2048], dtype=np.int32)
    wl = inputs.make_prefill_workload("p1", device="cpu", new=[1] * len(lens), prior=lens - 1,
                                      num_q_heads=32, num_kv_heads=8, seed=5).to("cuda")
    out, status = _gpu(psd, wl)
    assert status == 0
    ref = oracle.decode_attention(inputs.bf16_bits(wl.q), inputs.bf16_bits(wl.k_cache),
                                  inputs.bf16_bits(wl.v_cache), wl.block_table.cpu().numpy(), wl.lengths, 8,
                                  wl.scale)
    _compare(out, ref, "Q=1")
    attn = psd.DecodeAttention(len(lens), 32, 8, 128, 16, wl.block_table.shape[1], wl.k_cache.shape[0])
    dec = attn(wl.q, wl.k_cache, wl.v_cache, wl.block_table, wl.seq_lens, scale=wl.scale)
    torch.cuda.synchronize()
    attn.close()
    _compare(dec, ref, "decode")


def test_prefill_is_deterministic_and_blind_to_block_relabelling(psd):
    wl = inputs.make_prefill_workload("p1", device="cpu", new=[200, 90], prior=[300, 0], num_q_heads=32,
                                      num_kv_heads=8, spare_blocks=7, seed=9)
    g = wl.to("cuda")
    a, sa = _gpu(psd, g)
    b, sb = _gpu(psd, g)
    assert sa == sb == 0
    assert torch.equal(a, b)
    # Move every page to another physical block: same bits out.
    nb = wl.k_cache.shape[0]
    perm = np.random.default_rng(4).permutation(nb)
    k2 = torch.empty_like(wl.k_cache)
    v2 = torch.empty_like(wl.v_cache)
    k2[perm] = wl.k_cache
    v2[perm] = wl.v_cache
    bt = wl.block_table.numpy()
    bt2 = np.where(bt >= 0, perm[np.maximum(bt, 0)], -1).astype(np.int32)
    g2 = inputs.PrefillWorkload(cfg=wl.cfg, q=wl.q, k_cache=k2, v_cache=v2, block_table=torch.from_numpy(bt2),
                                seq_lens=wl.seq_lens, q_start=wl.q_start, q_lens=wl.q_lens, lengths=wl.lengths,
                                scale=wl.scale).to("cuda")
    c, sc = _gpu(psd, g2)
    assert sc == 0
    assert torch.equal(a, c)


def test_prefill_flags_bad_block_and_inconsistent_chunk(psd):
    wl = inputs.make_prefill_workload("p1", device="cpu", new=[40, 30], prior=[100, 10], num_q_heads=8,
                                      num_kv_heads=2, seed=3).to("cuda")
    bt_bad = wl.block_table.clone()
    bt_bad[0, 2] = wl.k_cache.shape[0] + 5
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    psd.prefill_attention(wl.q, wl.k_cache, wl.v_cache, bt_bad, wl.seq_lens, wl.q_start, wl.max_q_len,
                          scale=wl.scale, device_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) & psd.PS_DEVICE_BAD_BLOCK
    # A chunk longer than its sequence is skipped: its rows stay as they were.
    sl_bad = wl.seq_lens.clone()
    sl_bad[1] = 20  # Q_1 = 30 > 20
    status.zero_()
    out = torch.full_like(wl.q, 3.0)
    psd.prefill_attention(wl.q, wl.k_cache, wl.v_cache, wl.block_table, sl_bad, wl.q_start, wl.max_q_len,
                          out=out, scale=wl.scale, device_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) & psd.PS_DEVICE_LEN_CLAMPED
    assert torch.all(out[40:] == 3.0)
    ref = _oracle(wl)
    _compare(out[:40], ref[:40], "valid sequence next to a skipped one")


def test_prefill_rejects_bad_arguments(psd):
    wl = inputs.make_prefill_workload("p1", device="cpu", new=[5], prior=[5]).to("cuda")
    out = torch.empty_like(wl.q)
    args = [wl.q, wl.k_cache, wl.v_cache, wl.block_table, wl.seq_lens, wl.q_start, out, 1, 5, 5, 8, 2, 128, 16,
            wl.block_table.shape[1], wl.k_cache.shape[0], wl.scale, None, None]
    bad_dim = list(args)
    bad_dim[12] = 64
    with pytest.raises(psd.PsError):
        psd.ps_prefill_attention(*bad_dim)
    bad_group = list(args)
    bad_group[11] = 3  # 8 q heads over 3 kv heads
    with pytest.raises(psd.PsError):
        psd.ps_prefill_attention(*bad_group)
    bad_bs = list(args)
    bad_bs[13] = 8
    with pytest.raises(psd.PsError):
        psd.ps_prefill_attention(*bad_bs)
    bad_scale = list(args)
    bad_scale[16] = float("nan")
    with pytest.raises(psd.PsError):
        psd.ps_prefill_attention(*bad_scale)
    psd.ps_prefill_attention(*args)
    torch.cuda.synchronize()


def test_full_size_prefill_every_row(psd):
    """The 8-sequence Llama-3-8B chunked-prefill batch at full size, in the
    launch the bench times, against the prefill oracle on every output."""
    wl = inputs.make_prefill_workload("p2", device="cuda")
    out, status = _gpu(psd, wl)
    assert status == 0
    _compare(out, _oracle(wl), "p2, all %d outputs" % out.numel(), rel=0.0)


def test_full_size_prefill_runs_are_bit_identical(psd):
    """The kernel is deterministic (fixed tile order, fixed reduction order),
    so repeated launches of the full-size batch give the same bits; a race
    between the pipeline roles (a barrier wait passing on a stale phase, an
    accumulator read before its last P V) shows up as runs that differ."""
    wl = inputs.make_prefill_workload("p2", device="cuda")
    first, status = _gpu(psd, wl)
    assert status == 0
    for i in range(12):
        again, status = _gpu(psd, wl)
        assert status == 0
        assert torch.equal(again, first), "run %d differs from the first" % (i + 1)


def test_prefill_short_units_persistent(psd):
    """400 short chunks on short contexts (one to three 128-key tiles per
    unit): persistent clusters whose units leave one softmax group with no
    tile or a single one, every output against the oracle."""
    rng = np.random.default_rng(41)
    new = rng.integers(1, 65, size=400)
    prior = rng.integers(0, 201, size=400)
    wl = inputs.make_prefill_workload("p1", device="cpu", new=new, prior=prior, num_q_heads=32, num_kv_heads=8,
                                      seed=41).to("cuda")
    assert wl.seq_lens.shape[0] * 8 * ((wl.max_q_len + 31) // 32 + 1) // 2 <= 16384
    out, status = _gpu(psd, wl)
    assert status == 0
    _compare(out, _oracle(wl), "400 short chunks")


def test_prefill_with_more_units_than_a_persistent_launch_holds(psd):
    """Above 16384 units (sequence x KV head x pair of query tiles) the kernel
    runs one unit per cluster instead of persistent clusters: 2100 short
    chunks x 8 KV heads (16800 units), every output against the oracle."""
    rng = np.random.default_rng(31)
    new = rng.integers(1, 33, size=2100)  # one query-tile pair per sequence at g = 4
    prior = rng.integers(0, 60, size=2100)
    wl = inputs.make_prefill_workload("p1", device="cpu", new=new, prior=prior, num_q_heads=32, num_kv_heads=8,
                                      seed=31).to("cuda")
    assert wl.seq_lens.shape[0] * 8 * ((wl.max_q_len + 31) // 32 + 1) // 2 > 16384
    out, status = _gpu(psd, wl)
    assert status == 0
    _compare(out, _oracle(wl), "16800 units")


def test_prefill_counts_one_launch_per_call(psd):
    wl = inputs.make_prefill_workload("p1", device="cpu", new=[50, 20], prior=[10, 300]).to("cuda")
    before = psd.ps_decode_launch_count()
    _gpu(psd, wl)
    _gpu(psd, wl)
    assert psd.ps_decode_launch_count() - before == 2


def test_long_prompt_chunk_every_row(psd):
    """One 8192-token chunk over 4096 cached tokens (128 query tiles of
    Llama-3-8B heads): every row against the prefill oracle, and sampled
    rows also as decode rows of the truncated context (the decode oracle)."""
    wl = inputs.make_prefill_workload("p2", device="cuda", new=[8192], prior=[4096])
    out, status = _gpu(psd, wl)
    assert status == 0
    _compare(out, _oracle(wl), "8192-token chunk, all rows", rel=0.0)
    rows = sorted({0, 1, 31, 32, 4095, 8191} | set(np.random.default_rng(3).integers(0, 8192, size=10).tolist()))
    ref = oracle.decode_attention(inputs.bf16_bits(wl.q[rows]), inputs.bf16_bits(wl.k_cache), inputs.bf16_bits(wl.v_cache),
                                  wl.block_table.cpu().numpy()[[0] * len(rows)],
                                  np.asarray([4096 + i + 1 for i in rows], dtype=np.int32), wl.k_cache.shape[1], wl.scale)
    got = out[rows].float().cpu().numpy().astype(np.float64)
    err = np.abs(got - ref)
    assert err.max() <= MAX_ABS, err.max()
    assert err.mean() <= MEAN_ABS, err.mean()


def test_prefill_flags_a_chunk_longer_than_max_q_len(psd):
    wl = inputs.make_prefill_workload("p1", device="cpu", new=[100, 20], prior=[30, 5], num_q_heads=8,
                                      num_kv_heads=2, seed=12).to("cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = torch.full_like(wl.q, 5.0)
    psd.prefill_attention(wl.q, wl.k_cache, wl.v_cache, wl.block_table, wl.seq_lens, wl.q_start, 40, out=out,
                          scale=wl.scale, device_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) & psd.PS_DEVICE_LEN_CLAMPED
    ref = _oracle(wl)
    # Rows inside the grid are right; the first sequence's rows past the
    # grid (tiles of 32 tokens: rows 64..99) are untouched.
    _compare(out[:64], ref[:64], "rows inside the grid")
    _compare(out[100:], ref[100:], "second sequence")
    assert torch.all(out[64:100] == 5.0)
