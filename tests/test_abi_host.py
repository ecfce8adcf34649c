"""Host-side checks of the C ABI (no GPU needed).

The library must load, export every function include/ps_decode.h declares,
reject bad arguments before touching the device, and size plans and
workspaces as documented.  No call here launches a kernel.
"""
import ctypes

import pytest

from paper_2608_21719_gb300 import build as _build

_build.build()
from paper_2608_21719_gb300 import ps_decode as psd  # noqa: E402


def test_every_declared_symbol_is_exported():
    names = psd.header_functions()
    expected = {"ps_decode_plan_create", "ps_decode_plan_create_ex", "ps_decode_plan_set_workspace",
                "ps_decode_plan_bind", "ps_decode_plan_destroy", "ps_decode_plan_info", "ps_decode_attention",
                "ps_decode_attention_planned", "ps_decode_append_attention_planned",
                "ps_decode_plan_set_timing_events",
                "ps_decode_plan_read_device_status", "ps_decode_launch_count", "ps_status_string",
                "ps_decode_abi_version", "ps_decode_attention_noalloc", "ps_kv_pack", "ps_kv_unpack",
                "ps_test_inject"}
    assert expected <= set(names)
    lib = ctypes.CDLL(psd.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), n


def test_binding_constants_match_the_header():
    text = open(psd.HEADER_PATH).read()
    assert "#define PS_NOALLOC_SCRATCH_BYTES (16u << 20)" in text
    assert psd.PS_NOALLOC_SCRATCH_BYTES == 16 << 20


def test_status_strings_and_version():
    assert psd.ps_status_string(0) == "ok"
    for s in (-1, -2, -3, -4, -5):
        assert psd.ps_status_string(s) not in ("ok", "unknown status")
    assert psd.ps_status_string(-99) == "unknown status"
    assert psd.ps_decode_abi_version() == 100


def _plan(**kw):
    args = dict(num_seqs=64, num_q_heads=32, num_kv_heads=8, head_dim=128, block_size=16, max_blocks_per_seq=256,
                num_blocks=12000, num_sms=152, max_workers=0, min_stages_per_worker=0)
    args.update(kw)
    return psd.ps_decode_plan_create_ex(**args)


def test_plan_sizing_matches_layout():
    plan, ws = _plan()
    try:
        info = psd.ps_decode_plan_info(plan)
        assert info["grid_ctas"] == 152
        W = 152 * info["workers_per_cta"]
        assert info["max_workers"] == W
        # header + per-segment counters (S x Hkv ints) + two partial slots per worker range,
        # 8 heads x (128 acc + m, l) fp32 each
        slots = 2 * W
        expect = 256 + 64 * 8 * 4 + slots * 8 * 128 * 4 + slots * 8 * 2 * 4
        assert ws == info["workspace_bytes"]
        assert expect <= ws <= expect + 4 * 256
        assert info["smem_bytes"] <= 227 * 1024
    finally:
        psd.ps_decode_plan_destroy(plan)


def test_max_seqs_plan_fits_shared_memory():
    plan, ws = _plan(num_seqs=4096)
    try:
        assert psd.ps_decode_plan_info(plan)["smem_bytes"] <= 227 * 1024
    finally:
        psd.ps_decode_plan_destroy(plan)


@pytest.mark.parametrize("kw,status", [
    (dict(num_seqs=0), psd.PS_ERR_INVALID_ARG),
    (dict(num_q_heads=30, num_kv_heads=8), psd.PS_ERR_INVALID_ARG),
    (dict(head_dim=64), psd.PS_ERR_UNSUPPORTED),
    (dict(num_q_heads=128, num_kv_heads=8), psd.PS_ERR_UNSUPPORTED),
    (dict(block_size=8), psd.PS_ERR_UNSUPPORTED),
    (dict(block_size=24), psd.PS_ERR_UNSUPPORTED),
    (dict(num_seqs=4097), psd.PS_ERR_UNSUPPORTED),
    (dict(num_blocks=0), psd.PS_ERR_INVALID_ARG),
    (dict(num_sms=-1), psd.PS_ERR_INVALID_ARG),
    (dict(num_sms=4097), psd.PS_ERR_UNSUPPORTED),  # the split's 32-bit arithmetic needs < 2^15 workers
    # 4096 sequences x 8 heads x 65536 tiles: tile and cost-unit counts past 2^31
    (dict(num_seqs=4096, num_kv_heads=8, num_q_heads=64, max_blocks_per_seq=65536), psd.PS_ERR_UNSUPPORTED),
])
def test_plan_rejects_bad_shapes(kw, status):
    with pytest.raises(psd.PsError) as ei:
        _plan(**kw)
    assert ei.value.status == status


def test_noalloc_rejects_what_the_planned_path_rejects():
    """The workspace-free entry point applies the planned path's shape check,
    including the 32-bit bound on the split's cost units: 4096 sequences x 8
    kv heads x 65535 tiles stay below 2^31 tiles, but the boundary weight of
    the 32768 segments pushes the units past it.  Both entry points reject
    it before any CUDA call."""
    S, Hkv, mbps = 4096, 8, 65535
    tiles = S * Hkv * mbps
    assert tiles < 2**31 <= tiles + 4 * Hkv * S
    with pytest.raises(psd.PsError) as ei:
        _plan(num_seqs=S, num_q_heads=8 * Hkv, num_kv_heads=Hkv, max_blocks_per_seq=mbps)
    assert ei.value.status == psd.PS_ERR_UNSUPPORTED
    with pytest.raises(psd.PsError) as ei:
        psd.ps_decode_attention_noalloc(256, 256, 256, 256, 256, 256, S, 8 * Hkv, Hkv, 128, 16, mbps, 1, 0.1, None)
    assert ei.value.status == psd.PS_ERR_UNSUPPORTED
    # The rest of the shared check: bad group, block size, head_dim, sequence count.
    for args, status in [((8, 3, 128, 16), psd.PS_ERR_INVALID_ARG), ((8, 2, 128, 8), psd.PS_ERR_UNSUPPORTED),
                         ((8, 2, 64, 16), psd.PS_ERR_UNSUPPORTED), ((128, 8, 128, 16), psd.PS_ERR_UNSUPPORTED)]:
        Hq, Hk, d, bs = args
        with pytest.raises(psd.PsError) as ei:
            psd.ps_decode_attention_noalloc(256, 256, 256, 256, 256, 256, 4, Hq, Hk, d, bs, 8, 100, 0.1, None)
        assert ei.value.status == status
    with pytest.raises(psd.PsError) as ei:
        psd.ps_decode_attention_noalloc(256, 256, 256, 256, 256, 256, 4097, 8, 2, 128, 16, 8, 100, 0.1, None)
    assert ei.value.status == psd.PS_ERR_UNSUPPORTED
    # Counters alone beyond the fixed array: 4096 sequences x 1025 kv heads x 4 bytes.
    assert 4096 * 1025 * 4 > psd.PS_NOALLOC_SCRATCH_BYTES
    with pytest.raises(psd.PsError) as ei:
        psd.ps_decode_attention_noalloc(256, 256, 256, 256, 256, 256, 4096, 1025, 1025, 128, 16, 1, 16, 0.1, None)
    assert ei.value.status == psd.PS_ERR_UNSUPPORTED


def test_calls_validate_before_touching_the_device():
    plan, ws = _plan()
    try:
        # no workspace yet
        with pytest.raises(psd.PsError) as ei:
            psd.ps_decode_attention_planned(plan, 16, 16, 16, 16, 16, 16, 0.1, None)
        assert ei.value.status == psd.PS_ERR_WORKSPACE
        # null / misaligned pointers
        with pytest.raises(psd.PsError) as ei:
            psd.ps_decode_attention_planned(plan, 0, 16, 16, 16, 16, 16, 0.1, None)
        assert ei.value.status == psd.PS_ERR_INVALID_ARG
        with pytest.raises(psd.PsError) as ei:
            psd.ps_decode_attention_planned(plan, 8, 16, 16, 16, 16, 16, 0.1, None)
        assert ei.value.status == psd.PS_ERR_INVALID_ARG
        with pytest.raises(psd.PsError) as ei:
            psd.ps_decode_attention_planned(plan, 16, 16, 16, 16, 16, 16, float("nan"), None)
        assert ei.value.status == psd.PS_ERR_INVALID_ARG
        # workspace too small / misaligned
        with pytest.raises(psd.PsError) as ei:
            psd.ps_decode_plan_set_workspace(plan, 256, ws - 1)
        assert ei.value.status == psd.PS_ERR_WORKSPACE
        with pytest.raises(psd.PsError) as ei:
            psd.ps_decode_plan_set_workspace(plan, 128, ws)
        assert ei.value.status == psd.PS_ERR_INVALID_ARG
    finally:
        psd.ps_decode_plan_destroy(plan)


def test_stream_binding_lookup():
    plan, ws = _plan()
    try:
        fake_stream = 0x1234
        # nothing bound to this stream
        with pytest.raises(psd.PsError) as ei:
            psd.ps_decode_attention(16, 16, 16, 16, 16, 16, 64, 32, 8, 128, 16, 0.1, fake_stream)
        assert ei.value.status == psd.PS_ERR_NO_PLAN
        psd.ps_decode_plan_bind(plan, fake_stream)
        # bound, but the dims differ from the plan
        with pytest.raises(psd.PsError) as ei:
            psd.ps_decode_attention(16, 16, 16, 16, 16, 16, 64, 32, 8, 128, 32, 0.1, fake_stream)
        assert ei.value.status == psd.PS_ERR_NO_PLAN
        # bound and matching, but no workspace: fails before any CUDA call
        with pytest.raises(psd.PsError) as ei:
            psd.ps_decode_attention(16, 16, 16, 16, 16, 16, 64, 32, 8, 128, 16, 0.1, fake_stream)
        assert ei.value.status == psd.PS_ERR_WORKSPACE
        psd.ps_decode_plan_bind(None, fake_stream)
        with pytest.raises(psd.PsError) as ei:
            psd.ps_decode_attention(16, 16, 16, 16, 16, 16, 64, 32, 8, 128, 16, 0.1, fake_stream)
        assert ei.value.status == psd.PS_ERR_NO_PLAN
        psd.ps_decode_plan_bind(plan, fake_stream)
    finally:
        psd.ps_decode_plan_destroy(plan)
    # destroying the plan dropped its binding
    with pytest.raises(psd.PsError) as ei:
        psd.ps_decode_attention(16, 16, 16, 16, 16, 16, 64, 32, 8, 128, 16, 0.1, 0x1234)
    assert ei.value.status == psd.PS_ERR_NO_PLAN


def test_worker_overrides_are_recorded():
    plan, _ = _plan(max_workers=1, min_stages_per_worker=3)
    try:
        info = psd.ps_decode_plan_info(plan)
        assert info["max_workers"] == 1 and info["min_stages_per_worker"] == 3
    finally:
        psd.ps_decode_plan_destroy(plan)


def test_kv_transfer_validates_on_the_host():
    off = 16
    with pytest.raises(psd.PsError) as ei:  # null pointer
        psd.ps_kv_pack(0, 16, 16, 4, 16, 2, 8, 128, 16, 100, off, 16, None, None)
    assert ei.value.status == psd.PS_ERR_INVALID_ARG
    with pytest.raises(psd.PsError) as ei:  # misaligned cache
        psd.ps_kv_pack(8, 16, 16, 4, 16, 2, 8, 128, 16, 100, off, 16, None, None)
    assert ei.value.status == psd.PS_ERR_INVALID_ARG
    with pytest.raises(psd.PsError) as ei:  # head_dim not a multiple of 8
        psd.ps_kv_unpack(16, off, 16, 4, 16, 2, 8, 100, 16, 100, 16, 16, None, None)
    assert ei.value.status == psd.PS_ERR_UNSUPPORTED
    with pytest.raises(psd.PsError) as ei:  # too many sequences
        psd.ps_kv_unpack(16, off, 16, 4, 16, 5000, 8, 128, 16, 100, 16, 16, None, None)
    assert ei.value.status == psd.PS_ERR_UNSUPPORTED


def test_fault_injection_arguments():
    for kind, value in [(0, 1), (4, 1), (psd.PS_INJECT_LAUNCH_ERROR, -1), (psd.PS_INJECT_LAUNCH_ERROR, 10001),
                        (psd.PS_INJECT_DECODE_STALL, 999), (psd.PS_INJECT_DECODE_STALL, 2 * 10**9),
                        (psd.PS_INJECT_PREFILL_STALL, 999), (psd.PS_INJECT_PREFILL_STALL, 2 * 10**9)]:
        with pytest.raises(psd.PsError) as ei:
            psd.ps_test_inject(kind, value)
        assert ei.value.status == psd.PS_ERR_INVALID_ARG
    # valid values, then cleared again so that nothing leaks into later calls
    psd.ps_test_inject(psd.PS_INJECT_LAUNCH_ERROR, 1)
    psd.ps_test_inject(psd.PS_INJECT_LAUNCH_ERROR, 0)
    psd.ps_test_inject(psd.PS_INJECT_DECODE_STALL, 10**6)
    psd.ps_test_inject(psd.PS_INJECT_DECODE_STALL, 0)
    psd.ps_test_inject(psd.PS_INJECT_PREFILL_STALL, 10**6)
    psd.ps_test_inject(psd.PS_INJECT_PREFILL_STALL, 0)


def test_prefill_validates_on_the_host():
    # Stand-in 16-byte-aligned device addresses: every case below is decided
    # before the call encodes a tensor map or touches the device.
    A = 256
    base = [A, A, A, A, A, A, A, 1, 5, 5, 8, 2, 128, 16, 4, 16, 0.1, None, None]

    def status(**changes):
        args = list(base)
        names = ["q", "k", "v", "bt", "sl", "qs", "out", "num_seqs", "total", "max_q", "hq", "hkv", "hd", "bs",
                 "mbps", "nb", "scale", "dev_status", "stream"]
        for k, v in changes.items():
            args[names.index(k)] = v
        try:
            psd.ps_prefill_attention(*args)
        except psd.PsError as e:
            return e.status
        return psd.PS_OK

    inval, unsup = psd.PS_ERR_INVALID_ARG, psd.PS_ERR_UNSUPPORTED
    assert status(q=0) == inval
    assert status(out=A + 8) == inval            # bf16 rows need 16-byte alignment
    assert status(bt=A + 2) == inval             # int32 arrays need 4-byte alignment
    assert status(dev_status=A + 1) == inval
    assert status(num_seqs=-1) == inval
    assert status(max_q=6) == inval              # above total_q_tokens
    assert status(hq=8, hkv=3) == inval          # heads not a multiple
    assert status(nb=0) == inval
    assert status(scale=float("inf")) == inval
    assert status(hd=64) == unsup
    assert status(hq=34, hkv=2) == unsup         # g = 17
    assert status(bs=8) == unsup                 # not a multiple of 16
    assert status(num_seqs=65536) == unsup
    assert status(total=10 ** 7, max_q=10 ** 7, hq=2, hkv=2) == unsup  # more than 65535 query tiles
    # nothing to do: no launch, no device call, PS_OK
    assert status(num_seqs=0) == psd.PS_OK
    assert status(total=0, max_q=0) == psd.PS_OK
    assert status(max_q=0) == psd.PS_OK
