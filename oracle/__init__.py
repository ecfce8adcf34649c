"""fp64 CPU oracle for paged GQA decode attention (test infrastructure only).

The compute lives in ``ps_oracle.c`` (plain C, pthreads, double precision);
this module only compiles it with gcc and marshals numpy arrays into it.
Only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  It shares nothing with the CUDA
library: no header, no helper, no constant.

What the oracle computes is documented at the top of ``ps_oracle.c``: the
decode-step attention of PowerSlider Sec. 2.2 over a block-table-paged KV
cache, in the KV layout ``[num_blocks][num_kv_heads][block_size][head_dim]``,
plus the causal chunked-prefill form over the same cache and the KV hand-off
pack/unpack gather and scatter.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "ps_oracle.c")
_LIB = os.path.join(_HERE, "libps_oracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False, src: str = _SRC, out: str = _LIB) -> str:
    """Compile the oracle shared library with gcc; returns the .so path."""
    if force or not os.path.exists(out) or os.path.getmtime(out) < os.path.getmtime(src):
        tmp = out + ".tmp%d" % os.getpid()
        cmd = ["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-pthread", "-o", tmp, src, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, out)
    return out


def _bind(path: str):
    lib = ctypes.CDLL(path)
    p = ctypes.c_void_p
    i = ctypes.c_int
    common = [p, p, p, p, p, i, i, i, i, i, i, ctypes.c_longlong, ctypes.c_double]
    lib.ps_oracle_decode_attention.argtypes = common + [i, p]
    lib.ps_oracle_decode_attention.restype = i
    lib.ps_oracle_decode_attention_split.argtypes = common + [i, i, p]
    lib.ps_oracle_decode_attention_split.restype = i
    lib.ps_oracle_prefill_attention.argtypes = [p, p, p, p, p, p, i, i, i, i, i, i, ctypes.c_longlong,
                                                ctypes.c_double, i, p]
    lib.ps_oracle_prefill_attention.restype = i
    lib.ps_oracle_kv_pack.argtypes = [p, p, p, i, p, i, i, i, i, ctypes.c_longlong, p, p]
    lib.ps_oracle_kv_pack.restype = i
    lib.ps_oracle_kv_unpack.argtypes = [p, p, p, i, p, i, i, i, i, ctypes.c_longlong, p, p]
    lib.ps_oracle_kv_unpack.restype = i
    return lib


def load(path: str | None = None):
    """Load (building if needed) the oracle library.  A custom path loads a
    separately compiled copy, which the mutation tests use."""
    global _lib
    if path is not None:
        return _bind(path)
    with _lock:
        if _lib is None:
            _lib = _bind(build())
    return _lib


ERRORS = {
    -1: "invalid argument",
    -2: "block id outside the pool",
    -3: "sequence longer than the block-table row",
    -4: "out of host memory",
}


def _as_u16(a) -> np.ndarray:
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint16:
        return a
    if a.dtype == np.int16:
        return a.view(np.uint16)
    raise TypeError("expected bfloat16 bit patterns as uint16/int16, got %s" % a.dtype)


def decode_attention(q_bits, k_bits, v_bits, block_table, seq_lens, num_kv_heads: int,
                     scale: float, num_blocks: int | None = None, chunk_tokens: int = 0,
                     num_threads: int | None = None, lib=None) -> np.ndarray:
    """fp64 decode attention.

    q_bits:      [S, Hq, d] bfloat16 bit patterns (uint16)
    k_bits/v_bits: [num_blocks, Hkv, bs, d] bfloat16 bit patterns (uint16)
    block_table: [S, max_blocks_per_seq] int32 (entries past a sequence's
                 last block are never read)
    seq_lens:    [S] int32
    chunk_tokens > 0 routes through the chunked log-sum-exp form.
    Returns out [S, Hq, d] float64.
    """
    lib = lib or load()
    q = _as_u16(q_bits)
    k = _as_u16(k_bits)
    v = _as_u16(v_bits)
    bt = np.ascontiguousarray(block_table, dtype=np.int32)
    sl = np.ascontiguousarray(seq_lens, dtype=np.int32)
    S, Hq, d = q.shape
    nb, hkv, bs, d2 = k.shape
    if v.shape != k.shape or d2 != d or hkv != num_kv_heads or bt.shape[0] != S or sl.shape != (S,):
        raise ValueError("inconsistent shapes")
    if num_blocks is None:
        num_blocks = nb
    out = np.empty((S, Hq, d), dtype=np.float64)
    threads = num_threads or os.cpu_count() or 1
    args = [q.ctypes.data, k.ctypes.data, v.ctypes.data, bt.ctypes.data, sl.ctypes.data,
            S, Hq, hkv, d, bs, bt.shape[1] if bt.ndim == 2 else 0, int(num_blocks), float(scale)]
    if chunk_tokens:
        rc = lib.ps_oracle_decode_attention_split(*args, int(chunk_tokens), int(threads), out.ctypes.data)
    else:
        rc = lib.ps_oracle_decode_attention(*args, int(threads), out.ctypes.data)
    if rc != 0:
        raise RuntimeError("oracle failed: %s (%d)" % (ERRORS.get(rc, "unknown"), rc))
    return out


def packed_offsets(seq_lens, num_kv_heads: int, head_dim: int) -> np.ndarray:
    """Element offsets of each sequence in a packed K/V hand-off buffer
    (sequence i takes 2 * Hkv * L_i * d elements)."""
    sizes = 2 * num_kv_heads * np.asarray(seq_lens, dtype=np.int64) * head_dim
    return np.concatenate([[0], np.cumsum(sizes)[:-1]]).astype(np.int64)


def kv_pack(k_bits, v_bits, block_table, seq_lens, offsets=None, lib=None) -> np.ndarray:
    """Gather each sequence's K/V pages into the packed hand-off layout
    [K: Hkv x L x d | V: Hkv x L x d] (bf16 bits, uint16)."""
    lib = lib or load()
    k = _as_u16(k_bits)
    v = _as_u16(v_bits)
    bt = np.ascontiguousarray(block_table, dtype=np.int32)
    sl = np.ascontiguousarray(seq_lens, dtype=np.int32)
    nb, hkv, bs, d = k.shape
    off = packed_offsets(sl, hkv, d) if offsets is None else np.ascontiguousarray(offsets, dtype=np.int64)
    total = int(off[-1] + 2 * hkv * int(sl[-1]) * d) if len(sl) else 0
    dst = np.zeros(max(total, 1), dtype=np.uint16)
    rc = lib.ps_oracle_kv_pack(k.ctypes.data, v.ctypes.data, bt.ctypes.data, bt.shape[1], sl.ctypes.data, len(sl),
                               hkv, d, bs, nb, off.ctypes.data, dst.ctypes.data)
    if rc != 0:
        raise RuntimeError("oracle kv_pack failed: %s (%d)" % (ERRORS.get(rc, "unknown"), rc))
    return dst[:total]


def kv_unpack(packed, k_bits, v_bits, block_table, seq_lens, offsets=None, lib=None):
    """Scatter a packed hand-off buffer into copies of the given caches
    through block_table; returns (k, v) as uint16 arrays."""
    lib = lib or load()
    k = _as_u16(k_bits).copy()
    v = _as_u16(v_bits).copy()
    src = _as_u16(packed)
    bt = np.ascontiguousarray(block_table, dtype=np.int32)
    sl = np.ascontiguousarray(seq_lens, dtype=np.int32)
    nb, hkv, bs, d = k.shape
    off = packed_offsets(sl, hkv, d) if offsets is None else np.ascontiguousarray(offsets, dtype=np.int64)
    rc = lib.ps_oracle_kv_unpack(src.ctypes.data, off.ctypes.data, bt.ctypes.data, bt.shape[1], sl.ctypes.data,
                                 len(sl), hkv, d, bs, nb, k.ctypes.data, v.ctypes.data)
    if rc != 0:
        raise RuntimeError("oracle kv_unpack failed: %s (%d)" % (ERRORS.get(rc, "unknown"), rc))
    return k, v


def prefill_attention(q_bits, k_bits, v_bits, block_table, seq_lens, q_start, num_kv_heads: int, scale: float,
                      num_threads: int | None = None, lib=None) -> np.ndarray:
    """fp64 chunked-prefill attention.  q_bits [T, Hq, d] holds the new tokens
    of every sequence (sequence s owns rows q_start[s] .. q_start[s+1]); they
    are the last tokens of the seq_lens[s] cached ones and attend causally.
    Returns out [T, Hq, d] float64."""
    lib = lib or load()
    q = _as_u16(q_bits)
    k = _as_u16(k_bits)
    v = _as_u16(v_bits)
    bt = np.ascontiguousarray(block_table, dtype=np.int32)
    sl = np.ascontiguousarray(seq_lens, dtype=np.int32)
    qs = np.ascontiguousarray(q_start, dtype=np.int32)
    T, Hq, d = q.shape
    nb, hkv, bs, d2 = k.shape
    if v.shape != k.shape or d2 != d or hkv != num_kv_heads or qs.shape != (len(sl) + 1,) or qs[-1] != T:
        raise ValueError("inconsistent shapes")
    out = np.empty((T, Hq, d), dtype=np.float64)
    rc = lib.ps_oracle_prefill_attention(q.ctypes.data, k.ctypes.data, v.ctypes.data, bt.ctypes.data,
                                         sl.ctypes.data, qs.ctypes.data, len(sl), Hq, hkv, d, bs, bt.shape[1], nb,
                                         float(scale), int(num_threads or os.cpu_count() or 1), out.ctypes.data)
    if rc != 0:
        raise RuntimeError("oracle prefill failed: %s (%d)" % (ERRORS.get(rc, "unknown"), rc))
    return out
