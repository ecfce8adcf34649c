"""Error paths on the GPU, with the faults injected by the library's test
hook (ps_test_inject): a launch that reports a CUDA error, and a bounded
in-kernel wait that runs out on an mbarrier nothing arrives on.  Nothing here
faults, traps or hangs the device; every test checks that the next call on the
same context works and matches the oracle.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_21719_gb300 import inputs

pytestmark = pytest.mark.gpu

MAX_ABS = 8e-3
MEAN_ABS = 1e-3
CUDA_ERROR_INVALID_VALUE = 1


@pytest.fixture(scope="module")
def psd():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_21719_gb300 import build
    build.build()
    from paper_2608_21719_gb300 import ps_decode
    yield ps_decode
    ps_decode.ps_test_inject(ps_decode.PS_INJECT_LAUNCH_ERROR, 0)
    ps_decode.ps_test_inject(ps_decode.PS_INJECT_DECODE_STALL, 0)
    ps_decode.ps_test_inject(ps_decode.PS_INJECT_PREFILL_STALL, 0)


def _oracle(wl):
    return oracle.decode_attention(inputs.bf16_bits(wl.q), inputs.bf16_bits(wl.k_cache),
                                   inputs.bf16_bits(wl.v_cache), wl.block_table.cpu().numpy(),
                                   wl.seq_lens.cpu().numpy(), wl.num_kv_heads, wl.scale)


def _check(got, ref):
    err = np.abs(got.float().cpu().numpy().astype(np.float64) - ref)
    assert err.max() <= MAX_ABS and err.mean() <= MEAN_ABS, (err.max(), err.mean())


def _call(attn, wl, out=None):
    return attn(wl.q, wl.k_cache, wl.v_cache, wl.block_table, wl.seq_lens, out=out, scale=wl.scale)


def test_injected_launch_error_is_reported_and_the_next_call_works(psd):
    wl = inputs.make_workload(1, device="cuda", poison=True)
    attn = psd.DecodeAttention.for_workload(wl)
    before = psd.ps_decode_launch_count()
    psd.ps_test_inject(psd.PS_INJECT_LAUNCH_ERROR, CUDA_ERROR_INVALID_VALUE)
    with pytest.raises(psd.PsError) as ei:
        _call(attn, wl)
    assert ei.value.status == psd.PS_ERR_CUDA
    assert psd.ps_decode_launch_count() == before  # nothing was launched
    out = _call(attn, wl)
    torch.cuda.synchronize()
    assert attn.device_status() == 0
    _check(out, _oracle(wl))
    attn.close()


@pytest.mark.parametrize("persistent", [True, False])
def test_injected_prefill_stall_times_out_and_the_next_call_works(psd, persistent):
    """The MMA issuer of every CTA pair first waits 2 ms on an mbarrier that
    nothing arrives on: the wait runs out, both CTAs of every pair give up
    (each raises the other's abort flag), PS_DEVICE_TIMEOUT is set, the copies
    in flight land, tensor memory is freed and no output is written; the next
    call on the same context is normal and matches the oracle.  Both launch
    forms: persistent clusters, and one unit per cluster (above 16384 units)."""
    if persistent:
        wl = inputs.make_prefill_workload("p1", device="cpu", new=[300, 90, 1], prior=[500, 0, 40],
                                          num_q_heads=32, num_kv_heads=8, seed=5)
    else:
        rng = np.random.default_rng(31)
        wl = inputs.make_prefill_workload("p1", device="cpu", new=rng.integers(1, 33, size=2100),
                                          prior=rng.integers(0, 60, size=2100), num_q_heads=32, num_kv_heads=8,
                                          seed=31)
    wl = wl.to("cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    sentinel = torch.full_like(wl.q, 3.0)
    psd.ps_test_inject(psd.PS_INJECT_PREFILL_STALL, 2_000_000)
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    start.record()
    out = psd.prefill_attention(wl.q, wl.k_cache, wl.v_cache, wl.block_table, wl.seq_lens, wl.q_start,
                                wl.max_q_len, out=sentinel.clone(), scale=wl.scale, device_status=status)
    end.record()
    torch.cuda.synchronize()
    ms = start.elapsed_time(end)
    assert 1.9 <= ms < 1000.0, ms  # ran to the injected limit; the other waits gave up with it
    assert int(status.item()) & psd.PS_DEVICE_TIMEOUT
    assert torch.equal(out, sentinel)  # no MMA ran, so no row was written
    status.zero_()
    out = psd.prefill_attention(wl.q, wl.k_cache, wl.v_cache, wl.block_table, wl.seq_lens, wl.q_start,
                                wl.max_q_len, scale=wl.scale, device_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    ref = oracle.prefill_attention(inputs.bf16_bits(wl.q), inputs.bf16_bits(wl.k_cache),
                                   inputs.bf16_bits(wl.v_cache), wl.block_table.cpu().numpy(), wl.lengths,
                                   wl.q_start.cpu().numpy(), wl.k_cache.shape[1], wl.scale)
    err = np.abs(out.float().cpu().numpy().astype(np.float64) - ref)
    assert err.max() <= MAX_ABS + 2.0 ** -8 * np.abs(ref).max() and err.mean() <= MEAN_ABS, (err.max(), err.mean())


def test_injected_launch_error_on_prefill_and_kv_pack(psd):
    wl = inputs.make_prefill_workload("p1", device="cpu", new=[50, 20], prior=[10, 300]).to("cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    psd.ps_test_inject(psd.PS_INJECT_LAUNCH_ERROR, CUDA_ERROR_INVALID_VALUE)
    with pytest.raises(psd.PsError) as ei:
        psd.prefill_attention(wl.q, wl.k_cache, wl.v_cache, wl.block_table, wl.seq_lens, wl.q_start,
                              wl.max_q_len, scale=wl.scale, device_status=status)
    assert ei.value.status == psd.PS_ERR_CUDA
    out = psd.prefill_attention(wl.q, wl.k_cache, wl.v_cache, wl.block_table, wl.seq_lens, wl.q_start,
                                wl.max_q_len, scale=wl.scale, device_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0 and torch.all(torch.isfinite(out.float()))

    L = np.asarray([40, 20], dtype=np.int32)
    bs, Hkv = 16, 2
    nb = inputs.blocks_needed(L, bs) + 1
    bt = inputs.build_block_table(L, bs, 4, nb, np.random.default_rng(1))
    kv = inputs.make_tensors(4, Hkv, 128, bs, bt, L, nb, seed=2, device="cuda", poison=False)
    off = torch.from_numpy(oracle.packed_offsets(L, Hkv, 128)).cuda()
    dst = torch.zeros(int(2 * Hkv * L.sum() * 128), dtype=torch.int16, device="cuda")
    args = (kv.k_cache, kv.v_cache, kv.block_table, 4, kv.seq_lens, 2, Hkv, 128, bs, nb, off, dst, status, None)
    psd.ps_test_inject(psd.PS_INJECT_LAUNCH_ERROR, CUDA_ERROR_INVALID_VALUE)
    with pytest.raises(psd.PsError) as ei:
        psd.ps_kv_pack(*args)
    assert ei.value.status == psd.PS_ERR_CUDA
    assert torch.all(dst == 0)  # nothing ran
    psd.ps_kv_pack(*args)
    torch.cuda.synchronize()
    assert int(status.item()) == 0 and bool(torch.any(dst != 0))


@pytest.mark.parametrize("key", [1, 2])
def test_injected_stall_times_out_and_the_plan_recovers(psd, key):
    # Every streaming warp first waits 2 ms on an mbarrier that nothing
    # arrives on: the bounded wait runs out, the kernel raises
    # PS_DEVICE_TIMEOUT, lets its in-flight copies land and exits without
    # writing output.  The context stays usable; after the documented
    # recovery (hand the workspace to the plan again) the next call is right.
    wl = inputs.make_workload(key, device="cuda", poison=False)
    assert int(wl.seq_lens.min()) > 0
    attn = psd.DecodeAttention.for_workload(wl)
    sentinel = torch.full_like(wl.q, 3.0)
    psd.ps_test_inject(psd.PS_INJECT_DECODE_STALL, 2_000_000)
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    start.record()
    out = _call(attn, wl, out=sentinel.clone())
    end.record()
    torch.cuda.synchronize()
    assert start.elapsed_time(end) >= 1.9  # ms: the wait ran to its limit
    assert attn.device_status() & psd.PS_DEVICE_TIMEOUT
    assert torch.equal(out, sentinel)  # no output was written
    psd.ps_decode_plan_set_workspace(attn.plan, attn.workspace, attn.ws_bytes)
    out = _call(attn, wl)
    torch.cuda.synchronize()
    assert attn.device_status() == 0
    if key == 1:
        _check(out, _oracle(wl))
    else:
        again = _call(attn, wl)
        torch.cuda.synchronize()
        assert torch.equal(out, again) and torch.all(torch.isfinite(out.float()))
    attn.close()
    del wl
    torch.cuda.empty_cache()
