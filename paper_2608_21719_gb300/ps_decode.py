"""ctypes binding to libps_decode.so (include/ps_decode.h).

Argument marshalling only: every step of the computation runs in the CUDA
kernels behind the C ABI.  Importing this module raises if the library has
not been built; there is no CPU fallback.

The functions keep the C names.  Pointer arguments accept either a torch
tensor (its data_ptr() is passed) or a plain integer address; stream
arguments accept a torch.cuda.Stream, an integer handle or None (the legacy
default stream).  A non-OK status raises PsError.
"""
from __future__ import annotations

import ctypes
import os
import re

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libps_decode.so")
HEADER_PATH = os.path.join(os.path.dirname(_PKG), "include", "ps_decode.h")

if not os.path.exists(LIB_PATH):
    raise ImportError(
        "libps_decode.so is not built (expected at %s); build it with "
        "`python -m paper_2608_21719_gb300.build` or __graft_entry__.build()" % LIB_PATH)

_lib = ctypes.CDLL(LIB_PATH)

PS_OK = 0
PS_ERR_INVALID_ARG = -1
PS_ERR_UNSUPPORTED = -2
PS_ERR_NO_PLAN = -3
PS_ERR_WORKSPACE = -4
PS_ERR_CUDA = -5
PS_DEVICE_TIMEOUT = 1
PS_DEVICE_BAD_BLOCK = 2
PS_DEVICE_LEN_CLAMPED = 4
PS_INJECT_LAUNCH_ERROR = 1
PS_INJECT_DECODE_STALL = 2
PS_INJECT_PREFILL_STALL = 3
PS_NOALLOC_SCRATCH_BYTES = 16 << 20  # size of the workspace-free entry point's fixed device array


class PsError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__("%s: %s (%d)" % (where, ps_status_string(status), status))


class PlanInfo(ctypes.Structure):
    _fields_ = [
        ("num_seqs", ctypes.c_int), ("num_q_heads", ctypes.c_int), ("num_kv_heads", ctypes.c_int),
        ("head_dim", ctypes.c_int), ("block_size", ctypes.c_int), ("max_blocks_per_seq", ctypes.c_int),
        ("num_blocks", ctypes.c_longlong), ("num_sms", ctypes.c_int), ("grid_ctas", ctypes.c_int),
        ("workers_per_cta", ctypes.c_int), ("stages_per_worker", ctypes.c_int), ("max_workers", ctypes.c_int),
        ("min_stages_per_worker", ctypes.c_int), ("workspace_bytes", ctypes.c_size_t),
        ("smem_bytes", ctypes.c_size_t),
    ]

    def as_dict(self) -> dict:
        return {f: getattr(self, f) for f, _ in self._fields_}


_vp, _i, _sz, _f = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t, ctypes.c_float
_PLAN_DIMS = [_i, _i, _i, _i, _i, _i, ctypes.c_longlong]

_SIGS = {
    "ps_decode_plan_create": (_i, _PLAN_DIMS + [ctypes.POINTER(_vp), ctypes.POINTER(_sz)]),
    "ps_decode_plan_create_ex": (_i, _PLAN_DIMS + [_i, _i, _i, ctypes.POINTER(_vp), ctypes.POINTER(_sz)]),
    "ps_decode_plan_set_workspace": (_i, [_vp, _vp, _sz]),
    "ps_decode_plan_bind": (_i, [_vp, _vp]),
    "ps_decode_plan_destroy": (_i, [_vp]),
    "ps_decode_plan_info": (_i, [_vp, ctypes.POINTER(PlanInfo)]),
    "ps_decode_attention": (_i, [_vp, _vp, _vp, _vp, _vp, _vp, _i, _i, _i, _i, _i, _f, _vp]),
    "ps_decode_attention_planned": (_i, [_vp, _vp, _vp, _vp, _vp, _vp, _vp, _f, _vp]),
    "ps_decode_append_attention_planned": (_i, [_vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _f, _vp]),
    "ps_decode_plan_set_timing_events": (_i, [_vp, _vp, _vp]),
    "ps_decode_plan_read_device_status": (_i, [_vp, _vp, ctypes.POINTER(ctypes.c_uint)]),
    "ps_decode_attention_noalloc": (_i, [_vp, _vp, _vp, _vp, _vp, _vp, _i, _i, _i, _i, _i, _i, ctypes.c_longlong,
                                         _f, _vp]),
    "ps_kv_pack": (_i, [_vp, _vp, _vp, _i, _vp, _i, _i, _i, _i, ctypes.c_longlong, _vp, _vp, _vp, _vp]),
    "ps_kv_unpack": (_i, [_vp, _vp, _vp, _i, _vp, _i, _i, _i, _i, ctypes.c_longlong, _vp, _vp, _vp, _vp]),
    "ps_prefill_attention": (_i, [_vp, _vp, _vp, _vp, _vp, _vp, _vp, _i, _i, _i, _i, _i, _i, _i, _i,
                                  ctypes.c_longlong, _f, _vp, _vp]),
    "ps_decode_launch_count": (ctypes.c_ulonglong, []),
    "ps_test_inject": (_i, [_i, ctypes.c_longlong]),
    "ps_status_string": (ctypes.c_char_p, [_i]),
    "ps_decode_abi_version": (_i, []),
}
for _name, (_res, _args) in _SIGS.items():
    _fn = getattr(_lib, _name)
    _fn.restype = _res
    _fn.argtypes = _args


def header_functions(path: str = HEADER_PATH) -> list:
    """Names of every function declared in include/ps_decode.h."""
    text = re.sub(r"/\*.*?\*/", "", open(path).read(), flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[A-Za-z_][\w ]*?[\s\*]+(ps_\w+)\s*\(", text, flags=re.M)))


def _ptr(x) -> int | None:
    if x is None:
        return None
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    return int(x)


def _stream(s) -> int | None:
    if s is None:
        return None
    if hasattr(s, "cuda_stream"):
        return s.cuda_stream or None
    return int(s) or None


def _check(status: int, where: str) -> None:
    if status != PS_OK:
        raise PsError(status, where)


def ps_status_string(status: int) -> str:
    return _lib.ps_status_string(int(status)).decode()


def ps_decode_abi_version() -> int:
    return _lib.ps_decode_abi_version()


def ps_decode_launch_count() -> int:
    return _lib.ps_decode_launch_count()


def ps_test_inject(kind, value) -> None:
    _check(_lib.ps_test_inject(int(kind), int(value)), "ps_test_inject")


def ps_decode_plan_create(num_seqs, num_q_heads, num_kv_heads, head_dim, block_size, max_blocks_per_seq,
                          num_blocks):
    """Returns (plan handle, workspace bytes)."""
    plan, ws = _vp(), _sz()
    _check(_lib.ps_decode_plan_create(num_seqs, num_q_heads, num_kv_heads, head_dim, block_size,
                                      max_blocks_per_seq, num_blocks, ctypes.byref(plan), ctypes.byref(ws)),
           "ps_decode_plan_create")
    return plan.value, ws.value


def ps_decode_plan_create_ex(num_seqs, num_q_heads, num_kv_heads, head_dim, block_size, max_blocks_per_seq,
                             num_blocks, num_sms=0, max_workers=0, min_stages_per_worker=0):
    plan, ws = _vp(), _sz()
    _check(_lib.ps_decode_plan_create_ex(num_seqs, num_q_heads, num_kv_heads, head_dim, block_size,
                                         max_blocks_per_seq, num_blocks, num_sms, max_workers,
                                         min_stages_per_worker, ctypes.byref(plan), ctypes.byref(ws)),
           "ps_decode_plan_create_ex")
    return plan.value, ws.value


def ps_decode_plan_set_workspace(plan, workspace, nbytes) -> None:
    _check(_lib.ps_decode_plan_set_workspace(plan, _ptr(workspace), int(nbytes)), "ps_decode_plan_set_workspace")


def ps_decode_plan_bind(plan, stream) -> None:
    _check(_lib.ps_decode_plan_bind(plan, _stream(stream)), "ps_decode_plan_bind")


def ps_decode_plan_destroy(plan) -> None:
    _check(_lib.ps_decode_plan_destroy(plan), "ps_decode_plan_destroy")


def ps_decode_plan_info(plan) -> dict:
    info = PlanInfo()
    _check(_lib.ps_decode_plan_info(plan, ctypes.byref(info)), "ps_decode_plan_info")
    return info.as_dict()


def ps_decode_attention(q, k_cache, v_cache, block_table, seq_lens, out, num_seqs, num_q_heads, num_kv_heads,
                        head_dim, block_size, scale, stream) -> None:
    _check(_lib.ps_decode_attention(_ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(block_table), _ptr(seq_lens),
                                    _ptr(out), num_seqs, num_q_heads, num_kv_heads, head_dim, block_size,
                                    float(scale), _stream(stream)), "ps_decode_attention")


def ps_decode_attention_planned(plan, q, k_cache, v_cache, block_table, seq_lens, out, scale, stream) -> None:
    _check(_lib.ps_decode_attention_planned(plan, _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(block_table),
                                            _ptr(seq_lens), _ptr(out), float(scale), _stream(stream)),
           "ps_decode_attention_planned")


def ps_decode_append_attention_planned(plan, q, k_new, v_new, k_cache, v_cache, block_table, seq_lens, out,
                                       scale, stream) -> None:
    _check(_lib.ps_decode_append_attention_planned(plan, _ptr(q), _ptr(k_new), _ptr(v_new), _ptr(k_cache),
                                                   _ptr(v_cache), _ptr(block_table), _ptr(seq_lens), _ptr(out),
                                                   float(scale), _stream(stream)),
           "ps_decode_append_attention_planned")


def ps_decode_attention_noalloc(q, k_cache, v_cache, block_table, seq_lens, out, num_seqs, num_q_heads,
                                num_kv_heads, head_dim, block_size, max_blocks_per_seq, num_blocks, scale,
                                stream) -> None:
    """Decode attention with no plan and no workspace (scratch in a fixed
    device array inside the library; see include/ps_decode.h)."""
    _check(_lib.ps_decode_attention_noalloc(_ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(block_table),
                                            _ptr(seq_lens), _ptr(out), num_seqs, num_q_heads, num_kv_heads,
                                            head_dim, block_size, max_blocks_per_seq, num_blocks, float(scale),
                                            _stream(stream)), "ps_decode_attention_noalloc")


def ps_kv_pack(k_cache, v_cache, block_table, max_blocks_per_seq, seq_lens, num_seqs, num_kv_heads, head_dim,
               block_size, num_blocks, dst_offsets, dst, device_status, stream) -> None:
    _check(_lib.ps_kv_pack(_ptr(k_cache), _ptr(v_cache), _ptr(block_table), max_blocks_per_seq, _ptr(seq_lens),
                           num_seqs, num_kv_heads, head_dim, block_size, num_blocks, _ptr(dst_offsets), _ptr(dst),
                           _ptr(device_status), _stream(stream)), "ps_kv_pack")


def ps_kv_unpack(src, src_offsets, block_table, max_blocks_per_seq, seq_lens, num_seqs, num_kv_heads, head_dim,
                 block_size, num_blocks, k_cache, v_cache, device_status, stream) -> None:
    _check(_lib.ps_kv_unpack(_ptr(src), _ptr(src_offsets), _ptr(block_table), max_blocks_per_seq, _ptr(seq_lens),
                             num_seqs, num_kv_heads, head_dim, block_size, num_blocks, _ptr(k_cache), _ptr(v_cache),
                             _ptr(device_status), _stream(stream)), "ps_kv_unpack")


def ps_prefill_attention(q, k_cache, v_cache, block_table, seq_lens, q_start, out, num_seqs, total_q_tokens,
                         max_q_len, num_q_heads, num_kv_heads, head_dim, block_size, max_blocks_per_seq, num_blocks,
                         scale, device_status, stream) -> None:
    _check(_lib.ps_prefill_attention(_ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(block_table), _ptr(seq_lens),
                                     _ptr(q_start), _ptr(out), num_seqs, total_q_tokens, max_q_len, num_q_heads,
                                     num_kv_heads, head_dim, block_size, max_blocks_per_seq, num_blocks, scale,
                                     _ptr(device_status), _stream(stream)), "ps_prefill_attention")


def prefill_attention(q, k_cache, v_cache, block_table, seq_lens, q_start, max_q_len, out=None, scale=None,
                      device_status=None, stream=None):
    """Tensor-level wrapper: q [T, Hq, 128] bf16 on the GPU, caches
    [num_blocks, Hkv, bs, 128], block_table [S, mbps] int32, seq_lens [S]
    int32, q_start [S + 1] int32.  Returns out [T, Hq, 128] bf16."""
    import torch
    T, Hq, d = q.shape
    nb, hkv, bs, _ = k_cache.shape
    if out is None:
        out = torch.empty_like(q)
    if scale is None:
        scale = d ** -0.5
    ps_prefill_attention(q, k_cache, v_cache, block_table, seq_lens, q_start, out, seq_lens.shape[0], T,
                         int(max_q_len), Hq, hkv, d, bs, block_table.shape[1], nb, float(scale), device_status,
                         stream)
    return out


def ps_decode_plan_set_timing_events(plan, ev_start, ev_end) -> None:
    def h(e):
        if e is None:
            return None
        if hasattr(e, "cuda_event"):
            if not e.cuda_event:  # torch creates the CUDA event on its first record()
                e.record()
            return int(e.cuda_event)
        return int(e)
    _check(_lib.ps_decode_plan_set_timing_events(plan, h(ev_start), h(ev_end)),
           "ps_decode_plan_set_timing_events")


def ps_decode_plan_read_device_status(plan, stream) -> int:
    flags = ctypes.c_uint()
    _check(_lib.ps_decode_plan_read_device_status(plan, _stream(stream), ctypes.byref(flags)),
           "ps_decode_plan_read_device_status")
    return flags.value


class DecodeAttention:
    """Owns one plan and its workspace for a fixed batch shape.

    ``workload``-style tensors: q [S, Hq, 128] bf16, k/v caches
    [num_blocks, Hkv, bs, 128] bf16, block_table [S, mbps] int32,
    seq_lens [S] int32, all on one CUDA device.
    """

    def __init__(self, num_seqs, num_q_heads, num_kv_heads, head_dim, block_size, max_blocks_per_seq,
                 num_blocks, device=None, max_workers=0, min_stages_per_worker=0, num_sms=0):
        import torch
        self.plan, self.ws_bytes = ps_decode_plan_create_ex(
            num_seqs, num_q_heads, num_kv_heads, head_dim, block_size, max_blocks_per_seq, num_blocks,
            num_sms, max_workers, min_stages_per_worker)
        self.workspace = torch.empty(self.ws_bytes, dtype=torch.uint8, device=device or "cuda")
        ps_decode_plan_set_workspace(self.plan, self.workspace, self.ws_bytes)
        self.shape = (num_seqs, num_q_heads, num_kv_heads, head_dim, block_size)

    @classmethod
    def for_workload(cls, wl, **kw):
        return cls(wl.num_seqs, wl.num_q_heads, wl.num_kv_heads, wl.head_dim, wl.block_size,
                   wl.max_blocks_per_seq, wl.num_blocks, device=wl.q.device, **kw)

    def info(self) -> dict:
        return ps_decode_plan_info(self.plan)

    def __call__(self, q, k_cache, v_cache, block_table, seq_lens, out=None, scale=None, stream=None):
        import torch
        if out is None:
            out = torch.empty_like(q)
        if scale is None:
            scale = 1.0 / (q.shape[-1] ** 0.5)
        if stream is None:
            stream = torch.cuda.current_stream(q.device)
        ps_decode_attention_planned(self.plan, q, k_cache, v_cache, block_table, seq_lens, out, scale, stream)
        return out

    def append(self, q, k_new, v_new, k_cache, v_cache, block_table, seq_lens, out=None, scale=None, stream=None):
        """Append the current token's K/V to the cache and attend (one launch)."""
        import torch
        if out is None:
            out = torch.empty_like(q)
        if scale is None:
            scale = 1.0 / (q.shape[-1] ** 0.5)
        if stream is None:
            stream = torch.cuda.current_stream(q.device)
        ps_decode_append_attention_planned(self.plan, q, k_new, v_new, k_cache, v_cache, block_table, seq_lens,
                                           out, scale, stream)
        return out

    def device_status(self, stream=None) -> int:
        import torch
        return ps_decode_plan_read_device_status(self.plan, stream or torch.cuda.current_stream())

    def close(self):
        if self.plan:
            ps_decode_plan_destroy(self.plan)
            self.plan = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
