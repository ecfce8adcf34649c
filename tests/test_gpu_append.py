"""GPU parity of the fused append + decode attention step.

The reference is the definition: write the current token's K/V rows into
their cache slot on the host, then run the fp64 oracle on the updated cache.
The GPU call must give the same attention output (within the usual bounds)
and leave exactly the same cache bits (every other slot untouched).  The
target slot holds NaN before the call, so reading the stale slot instead of
k_new / v_new would show.
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


def _case(Hq, Hkv, bs, lengths, seed):
    lengths = np.asarray(lengths, dtype=np.int32)
    mbps = max(1, (int(lengths.max()) + bs - 1) // bs + 1)
    nb = inputs.blocks_needed(lengths, bs) + 4
    bt = inputs.build_block_table(lengths, bs, mbps, nb, np.random.default_rng(seed))
    wl = inputs.make_tensors(Hq, Hkv, 128, bs, bt, lengths, nb, seed, device="cpu")
    # The current token's slot is stale (NaN) until the append writes it.
    for s, L in enumerate(lengths):
        if L > 0:
            b = int(bt[s, (L - 1) // bs])
            wl.k_cache[b, :, (L - 1) % bs] = float("nan")
            wl.v_cache[b, :, (L - 1) % bs] = float("nan")
    gen = torch.Generator().manual_seed(seed + 99)
    k_new = torch.randn((len(lengths), Hkv, 128), generator=gen).to(torch.bfloat16)
    v_new = torch.randn((len(lengths), Hkv, 128), generator=gen).to(torch.bfloat16)
    return wl, k_new, v_new


def _host_append(wl, k_new, v_new):
    k = wl.k_cache.clone()
    v = wl.v_cache.clone()
    bs = wl.block_size
    for s, L in enumerate(wl.seq_lens.tolist()):
        if L > 0:
            b = int(wl.block_table[s, (L - 1) // bs])
            k[b, :, (L - 1) % bs] = k_new[s]
            v[b, :, (L - 1) % bs] = v_new[s]
    return k, v


def _run(psd, wl, k_new, v_new):
    g = wl.to("cuda")
    kn, vn = k_new.cuda(), v_new.cuda()
    attn = psd.DecodeAttention.for_workload(g)
    out = attn.append(g.q, kn, vn, g.k_cache, g.v_cache, g.block_table, g.seq_lens, scale=g.scale)
    torch.cuda.synchronize()
    status = attn.device_status()
    attn.close()
    return out.cpu(), g.k_cache.cpu(), g.v_cache.cpu(), status


def _check(out, ref, rel=BF16_REL):
    got = out.float().numpy().astype(np.float64)
    assert np.all(np.isfinite(got))
    err = np.abs(got - ref)
    assert np.all(err <= MAX_ABS + rel * np.abs(ref)), "max abs err %.3g" % err.max()
    assert err.mean() <= MEAN_ABS


@pytest.mark.parametrize("Hq,Hkv,bs,lengths", [
    (32, 8, 16, [1, 16, 17, 300, 1024, 0, 33]),
    (8, 2, 32, [5, 64, 65, 2000]),
    (64, 8, 16, [3000, 1, 511, 512, 513]),
    (4, 4, 64, [1, 63, 64, 65, 200]),
])
def test_append_matches_write_then_attend(psd, Hq, Hkv, bs, lengths):
    wl, k_new, v_new = _case(Hq, Hkv, bs, lengths, seed=len(lengths) * 7 + bs)
    k_ref, v_ref = _host_append(wl, k_new, v_new)
    ref = oracle.decode_attention(inputs.bf16_bits(wl.q), inputs.bf16_bits(k_ref), inputs.bf16_bits(v_ref),
                                  wl.block_table.numpy(), wl.seq_lens.numpy(), Hkv, wl.scale)
    out, k_gpu, v_gpu, status = _run(psd, wl, k_new, v_new)
    assert status == 0
    _check(out, ref)
    # The cache after the call: the appended rows, every other bit unchanged.
    assert torch.equal(k_gpu.view(torch.int16), k_ref.view(torch.int16))
    assert torch.equal(v_gpu.view(torch.int16), v_ref.view(torch.int16))
    for s, L in enumerate(lengths):
        if L == 0:
            assert torch.all(out[s] == 0)


def test_single_token_append_returns_the_new_value(psd):
    wl, k_new, v_new = _case(8, 2, 16, [1, 1, 1], seed=3)
    out, _, _, _ = _run(psd, wl, k_new, v_new)
    for s in range(3):
        for h in range(8):
            assert torch.equal(out[s, h], v_new[s, h // 4])


def test_append_at_full_size_every_output(psd):
    """The Llama-3-8B-shaped batch at full size: every output against the
    oracle on the host-appended cache, and the whole cache bit-for-bit."""
    wl = inputs.make_workload(2, device="cuda", poison=False)
    gen = torch.Generator(device="cuda").manual_seed(1234)
    k_new = torch.randn((wl.num_seqs, wl.num_kv_heads, 128), generator=gen, device="cuda").to(torch.bfloat16)
    v_new = torch.randn((wl.num_seqs, wl.num_kv_heads, 128), generator=gen, device="cuda").to(torch.bfloat16)
    host = inputs.Workload(cfg=None, q=wl.q.cpu(), k_cache=wl.k_cache.cpu(), v_cache=wl.v_cache.cpu(),
                           block_table=wl.block_table.cpu(), seq_lens=wl.seq_lens.cpu(), scale=wl.scale)
    k_ref, v_ref = _host_append(host, k_new.cpu(), v_new.cpu())
    attn = psd.DecodeAttention.for_workload(wl)
    out = attn.append(wl.q, k_new, v_new, wl.k_cache, wl.v_cache, wl.block_table, wl.seq_lens, scale=wl.scale)
    torch.cuda.synchronize()
    assert attn.device_status() == 0
    attn.close()
    assert torch.equal(wl.k_cache.cpu().view(torch.int16), k_ref.view(torch.int16))
    assert torch.equal(wl.v_cache.cpu().view(torch.int16), v_ref.view(torch.int16))
    ref = oracle.decode_attention(inputs.bf16_bits(host.q), inputs.bf16_bits(k_ref), inputs.bf16_bits(v_ref),
                                  host.block_table.numpy(), host.seq_lens.numpy(), wl.num_kv_heads, wl.scale)
    _check(out.cpu(), ref, rel=0.0)
