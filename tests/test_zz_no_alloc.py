"""The allocation-free entry point (GPU).

Callers that cannot allocate device memory -- a plugin whose host engine
owns every allocation, a foreign-function caller that only holds the
tensors it passes, a server that forbids allocation after start-up -- call
ps_decode_attention_noalloc, whose split-KV scratch is a fixed device array
inside the library.  These tests call it through the C ABI and check it
against the planned entry point, twice in a row, since the array keeps the
previous call's contents.  The split is the planned path's default one
(every streaming warp, the default minimum share), so the output must be
bit-identical to the planned call's; it is also held to the fp64 oracle's
bounds.  This file is collected last on purpose.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_21719_gb300 import inputs

pytestmark = pytest.mark.gpu

MAX_ABS = 8e-3
MEAN_ABS = 1e-3
BF16_REL = 2.0 ** -8  # bf16 output rounding, for short contexts with |o| > 1


@pytest.fixture(scope="module")
def psd():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_21719_gb300 import build
    build.build()
    from paper_2608_21719_gb300 import ps_decode
    return ps_decode


def _workload(Hq, Hkv, bs, lengths, seed):
    lengths = np.asarray(lengths, dtype=np.int32)
    mbps = max(1, (int(lengths.max()) + bs - 1) // bs + 1)
    nb = inputs.blocks_needed(lengths, bs) + 3
    bt = inputs.build_block_table(lengths, bs, mbps, nb, np.random.default_rng(seed))
    return inputs.make_tensors(Hq, Hkv, 128, bs, bt, lengths, nb, seed, device="cpu").to("cuda")


def _close(got, ref):
    got = got.float().cpu().numpy().astype(np.float64)
    assert np.all(np.isfinite(got))
    err = np.abs(got - ref)
    assert np.all(err <= MAX_ABS + BF16_REL * np.abs(ref)), "max abs err %.3g" % err.max()
    assert err.mean() <= MEAN_ABS


@pytest.mark.parametrize("case", [
    dict(Hq=32, Hkv=8, bs=16, lengths=[1, 200, 513, 16, 2049, 37, 777, 0, 64], seed=3),
    dict(Hq=64, Hkv=8, bs=32, lengths=[4000, 33, 1500, 9000], seed=4),
    dict(Hq=8, Hkv=2, bs=16, lengths=[37, 512, 100, 250], seed=5),
])
def test_noalloc_matches_planned_path_on_consecutive_calls(psd, case):
    wl = _workload(case["Hq"], case["Hkv"], case["bs"], case["lengths"], case["seed"])
    want = oracle.decode_attention(inputs.bf16_bits(wl.q), inputs.bf16_bits(wl.k_cache),
                                   inputs.bf16_bits(wl.v_cache), wl.block_table.cpu().numpy(),
                                   wl.seq_lens.cpu().numpy(), wl.num_kv_heads, wl.scale)
    attn = psd.DecodeAttention.for_workload(wl)
    ref = attn(wl.q, wl.k_cache, wl.v_cache, wl.block_table, wl.seq_lens, scale=wl.scale)
    torch.cuda.synchronize()
    attn.close()
    stream = torch.cuda.current_stream()
    for _ in range(2):
        out = torch.full_like(wl.q, float("nan"))
        psd.ps_decode_attention_noalloc(wl.q, wl.k_cache, wl.v_cache, wl.block_table, wl.seq_lens, out,
                                        wl.num_seqs, wl.num_q_heads, wl.num_kv_heads, 128, wl.block_size,
                                        wl.max_blocks_per_seq, wl.num_blocks, wl.scale, stream)
        torch.cuda.synchronize()
        assert torch.equal(out, ref)
        _close(out, want)


def test_noalloc_rejects_shapes_beyond_its_scratch(psd):
    # 4096 sequences x 1025 kv heads need 16.8 MB of per-segment counters
    # alone, more than the fixed array holds whatever the SM count, so the
    # call is rejected before anything is launched.
    assert 256 + 4096 * 1025 * 4 > psd.PS_NOALLOC_SCRATCH_BYTES
    t = torch.zeros(64, dtype=torch.int32, device="cuda")
    with pytest.raises(psd.PsError) as ei:
        psd.ps_decode_attention_noalloc(t, t, t, t, t, t, 4096, 1025, 1025, 128, 16, 1, 16, 0.1, None)
    assert ei.value.status == psd.PS_ERR_UNSUPPORTED
