"""GPU parity of the KV hand-off pack / unpack against the oracle (bit-exact).

pack must reproduce the oracle's packed buffer bit for bit; unpack into a
receiver pool (its own size and block permutation, NaN elsewhere) must give
the oracle's pool bit for bit, leaving every slot it does not own untouched.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_21719_gb300 import inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def psd():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_21719_gb300 import build
    build.build()
    from paper_2608_21719_gb300 import ps_decode
    return ps_decode


def _bits(t):
    return t.contiguous().cpu().view(torch.int16).numpy().view(np.uint16)


@pytest.mark.parametrize("Hkv,bs,lengths", [
    (8, 16, [1, 15, 16, 17, 300, 0, 1024]),
    (2, 32, [33, 64, 2000]),
    (8, 64, [4096, 1, 65]),
])
def test_pack_then_unpack_match_the_oracle(psd, Hkv, bs, lengths):
    L = np.asarray(lengths, dtype=np.int32)
    mbps = int(L.max()) // bs + 2
    nb = inputs.blocks_needed(L, bs) + 5
    bt = inputs.build_block_table(L, bs, mbps, nb, np.random.default_rng(3))
    wl = inputs.make_tensors(8, Hkv, 128, bs, bt, L, nb, seed=11, device="cpu", poison=True)
    off = oracle.packed_offsets(L, Hkv, 128)
    ref = oracle.kv_pack(inputs.bf16_bits(wl.k_cache), inputs.bf16_bits(wl.v_cache), bt, L, off)
    g = wl.to("cuda")
    off_d = torch.from_numpy(off).cuda()
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    dst = torch.full((max(1, ref.size),), -1, dtype=torch.int16, device="cuda")
    psd.ps_kv_pack(g.k_cache, g.v_cache, g.block_table, mbps, g.seq_lens, len(L), Hkv, 128, bs, nb, off_d, dst,
                   status, None)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    assert np.array_equal(_bits(dst)[:ref.size], ref)
    # Unpack into a receiver pool of another size and permutation.
    nb2 = inputs.blocks_needed(L, bs) + 11
    bt2 = inputs.build_block_table(L, bs, mbps, nb2, np.random.default_rng(8))
    k2 = torch.full((nb2, Hkv, bs, 128), float("nan"), dtype=torch.bfloat16)
    v2 = torch.full((nb2, Hkv, bs, 128), float("nan"), dtype=torch.bfloat16)
    k_ref, v_ref = oracle.kv_unpack(ref, inputs.bf16_bits(k2), inputs.bf16_bits(v2), bt2, L, off)
    k2d, v2d = k2.cuda(), v2.cuda()
    psd.ps_kv_unpack(dst, off_d, torch.from_numpy(bt2).cuda(), mbps, g.seq_lens, len(L), Hkv, 128, bs, nb2,
                     k2d, v2d, status, None)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    assert np.array_equal(_bits(k2d), k_ref)
    assert np.array_equal(_bits(v2d), v_ref)


def test_bad_block_is_skipped_and_flagged(psd):
    L = np.asarray([40, 20], dtype=np.int32)
    bs, Hkv = 16, 2
    nb = inputs.blocks_needed(L, bs) + 1
    bt = inputs.build_block_table(L, bs, 4, nb, np.random.default_rng(1))
    wl = inputs.make_tensors(4, Hkv, 128, bs, bt, L, nb, seed=2, device="cuda", poison=False)
    bt_bad = wl.block_table.clone()
    bt_bad[0, 1] = nb + 7
    off = torch.from_numpy(oracle.packed_offsets(L, Hkv, 128)).cuda()
    dst = torch.zeros(int(2 * Hkv * L.sum() * 128), dtype=torch.int16, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    before = psd.ps_decode_launch_count()
    psd.ps_kv_pack(wl.k_cache, wl.v_cache, bt_bad, 4, wl.seq_lens, 2, Hkv, 128, bs, nb, off, dst, status, None)
    torch.cuda.synchronize()
    assert psd.ps_decode_launch_count() - before == 1
    assert int(status.item()) & psd.PS_DEVICE_BAD_BLOCK
