"""Seeded synthetic workloads for paged GQA decode attention.

This module only builds inputs: sequence lengths, block tables over a
shuffled physical pool, and bf16 N(0, 1) query/key/value tensors.  It holds
none of the attention arithmetic, so both the CUDA path and the CPU oracle
can take their inputs from it.

The five named workloads stand in for the reasoning-serving mixes of
PowerSlider (Sec. 2.2: thinking chains are 10-100x longer than answers;
Sec. 3 Obs. 3: long heavy-tailed thinking contexts; Table 4 models
Llama-3-8B / Qwen-32B / Llama-70B shapes).  The paper's datasets (Magpie,
S1K, Azure traces) are not used; these length distributions replace them.

KV layout: ``[num_blocks][num_kv_heads][block_size][head_dim]`` bf16, so one
(block, kv-head) page of ``block_size * head_dim`` elements is contiguous.
Block table: int32 ``[num_seqs][max_blocks_per_seq]``, unused entries -1.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np
import torch

HEAD_DIM = 128


@dataclass(frozen=True)
class WorkloadConfig:
    key: int
    name: str
    num_seqs: int
    num_q_heads: int
    num_kv_heads: int
    block_size: int
    lengths: tuple  # ("uniform", lo, hi) | ("lognormal", median, sigma, lo, hi) | ("bimodal", ...)
    seed: int
    pool_blocks: int | None = None  # fixed pool size (else exactly the blocks needed)
    head_dim: int = HEAD_DIM
    max_len: int = field(default=0)

    @property
    def group(self) -> int:
        return self.num_q_heads // self.num_kv_heads


def _max_len(spec) -> int:
    kind = spec[0]
    if kind == "uniform":
        return spec[2]
    if kind == "lognormal":
        return spec[4]
    if kind == "bimodal":
        return max(spec[2][1], spec[3][1])
    raise ValueError(kind)


def _cfg(**kw) -> WorkloadConfig:
    c = WorkloadConfig(**kw)
    object.__setattr__(c, "max_len", _max_len(c.lengths))
    return c


# 6 GiB of K+V for the 70B-shaped workload: 32 tokens x 8 heads x 128 x 2 B x 2.
_POOL_6GIB_BS32_H8 = (6 << 30) // (32 * 8 * 128 * 2 * 2)

CONFIGS = {
    1: _cfg(key=1, name="tiny-gqa4", num_seqs=4, num_q_heads=8, num_kv_heads=2, block_size=16,
            lengths=("uniform", 37, 512), seed=0),
    2: _cfg(key=2, name="llama3-8b-decode", num_seqs=64, num_q_heads=32, num_kv_heads=8, block_size=16,
            lengths=("uniform", 1024, 4096), seed=1),
    3: _cfg(key=3, name="long-thinking-splitkv", num_seqs=16, num_q_heads=32, num_kv_heads=8, block_size=16,
            lengths=("lognormal", 12288, 0.5, 8192, 32768), seed=2),
    4: _cfg(key=4, name="mixed-phase-32b", num_seqs=128, num_q_heads=64, num_kv_heads=8, block_size=16,
            lengths=("bimodal", 0.4, (8192, 16384), (512, 2048)), seed=3),
    5: _cfg(key=5, name="70b-large-batch", num_seqs=256, num_q_heads=64, num_kv_heads=8, block_size=32,
            lengths=("uniform", 2048, 8192), seed=4, pool_blocks=_POOL_6GIB_BS32_H8),
}


def sample_lengths(cfg: WorkloadConfig, seed: int | None = None) -> np.ndarray:
    """Integer context lengths (current token included), inclusive ranges."""
    rng = np.random.default_rng(cfg.seed if seed is None else seed)
    spec = cfg.lengths
    S = cfg.num_seqs
    if spec[0] == "uniform":
        L = rng.integers(spec[1], spec[2], size=S, endpoint=True)
    elif spec[0] == "lognormal":
        _, median, sigma, lo, hi = spec
        L = np.rint(rng.lognormal(mean=math.log(median), sigma=sigma, size=S))
        L = np.clip(L, lo, hi)
    elif spec[0] == "bimodal":
        _, frac_long, (llo, lhi), (slo, shi) = spec
        n_long = int(round(frac_long * S))
        L = np.concatenate([rng.integers(llo, lhi, size=n_long, endpoint=True),
                            rng.integers(slo, shi, size=S - n_long, endpoint=True)])
        L = L[rng.permutation(S)]
    else:
        raise ValueError(spec[0])
    return L.astype(np.int32)


def blocks_needed(lengths: np.ndarray, block_size: int) -> int:
    return int(sum((int(l) + block_size - 1) // block_size for l in lengths))


def build_block_table(lengths: np.ndarray, block_size: int, max_blocks_per_seq: int,
                      num_blocks: int, rng: np.random.Generator) -> np.ndarray:
    """Assign each sequence's logical blocks to distinct, randomly permuted
    physical block ids of a pool of ``num_blocks``."""
    need = blocks_needed(lengths, block_size)
    if need > num_blocks:
        raise ValueError("pool too small: need %d blocks, have %d" % (need, num_blocks))
    perm = rng.permutation(num_blocks).astype(np.int32)
    bt = np.full((len(lengths), max_blocks_per_seq), -1, dtype=np.int32)
    pos = 0
    for s, l in enumerate(lengths):
        nb = (int(l) + block_size - 1) // block_size
        if nb > max_blocks_per_seq:
            raise ValueError("sequence %d needs %d blocks > row width %d" % (s, nb, max_blocks_per_seq))
        bt[s, :nb] = perm[pos:pos + nb]
        pos += nb
    return bt


@dataclass
class Workload:
    cfg: WorkloadConfig | None
    q: torch.Tensor            # [S, Hq, d] bf16
    k_cache: torch.Tensor      # [NB, Hkv, bs, d] bf16
    v_cache: torch.Tensor      # [NB, Hkv, bs, d] bf16
    block_table: torch.Tensor  # [S, mbps] int32
    seq_lens: torch.Tensor     # [S] int32
    scale: float

    def to(self, device) -> "Workload":
        return Workload(cfg=self.cfg, q=self.q.to(device), k_cache=self.k_cache.to(device),
                        v_cache=self.v_cache.to(device), block_table=self.block_table.to(device),
                        seq_lens=self.seq_lens.to(device), scale=self.scale)

    @property
    def num_seqs(self) -> int:
        return self.q.shape[0]

    @property
    def num_q_heads(self) -> int:
        return self.q.shape[1]

    @property
    def num_kv_heads(self) -> int:
        return self.k_cache.shape[1]

    @property
    def head_dim(self) -> int:
        return self.q.shape[2]

    @property
    def block_size(self) -> int:
        return self.k_cache.shape[2]

    @property
    def num_blocks(self) -> int:
        return self.k_cache.shape[0]

    @property
    def max_blocks_per_seq(self) -> int:
        return self.block_table.shape[1]


def poison_unused(k_cache: torch.Tensor, v_cache: torch.Tensor, block_table: np.ndarray,
                  lengths: np.ndarray) -> None:
    """Write NaN into every K/V slot that no sequence owns: spare blocks and
    the slots past the last token of each sequence's final block."""
    nb, _, bs, _ = k_cache.shape
    used = np.zeros(nb, dtype=bool)
    for s, l in enumerate(lengths):
        n = (int(l) + bs - 1) // bs
        used[block_table[s, :n]] = True
        tail = int(l) - (n - 1) * bs if n > 0 else bs
        if n > 0 and tail < bs:
            b = int(block_table[s, n - 1])
            k_cache[b, :, tail:, :] = float("nan")
            v_cache[b, :, tail:, :] = float("nan")
    spare = np.nonzero(~used)[0]
    if len(spare):
        idx = torch.from_numpy(spare).to(k_cache.device)
        k_cache.index_fill_(0, idx, float("nan"))
        v_cache.index_fill_(0, idx, float("nan"))


def make_workload(cfg: WorkloadConfig | int, device="cpu", poison: bool = True,
                  spare_blocks: int = 0, lengths: np.ndarray | None = None) -> Workload:
    """Build a named workload.  ``lengths`` overrides the sampled lengths
    (edge-case tests); ``spare_blocks`` adds unused (poisoned) pool blocks."""
    if isinstance(cfg, int):
        cfg = CONFIGS[cfg]
    seed = cfg.seed
    if lengths is None:
        lengths = sample_lengths(cfg, seed)
        if cfg.pool_blocks is not None:
            while blocks_needed(lengths, cfg.block_size) > cfg.pool_blocks:
                seed += 1
                lengths = sample_lengths(cfg, seed)
    lengths = np.asarray(lengths, dtype=np.int32)
    bs = cfg.block_size
    mbps = max(1, (max(cfg.max_len, int(lengths.max(initial=0))) + bs - 1) // bs)
    need = blocks_needed(lengths, bs)
    num_blocks = cfg.pool_blocks if cfg.pool_blocks is not None else need + spare_blocks
    num_blocks = max(num_blocks, 1)
    rng = np.random.default_rng(seed + 1000)
    bt = build_block_table(lengths, bs, mbps, num_blocks, rng)
    return make_tensors(cfg.num_q_heads, cfg.num_kv_heads, cfg.head_dim, bs, bt, lengths,
                        num_blocks, seed, device, poison, cfg)


def make_tensors(num_q_heads: int, num_kv_heads: int, head_dim: int, block_size: int,
                 block_table: np.ndarray, lengths: np.ndarray, num_blocks: int, seed: int,
                 device="cpu", poison: bool = True, cfg: WorkloadConfig | None = None) -> Workload:
    """Draw Q and the K/V pool as bf16 N(0, 1) from one seeded torch generator."""
    device = torch.device(device)
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed))
    S = len(lengths)
    q = torch.randn((S, num_q_heads, head_dim), generator=gen, device=device, dtype=torch.float32)
    q = q.to(torch.bfloat16)
    shape = (num_blocks, num_kv_heads, block_size, head_dim)
    k = torch.empty(shape, device=device, dtype=torch.bfloat16)
    v = torch.empty(shape, device=device, dtype=torch.bfloat16)
    # Fill in slabs so the fp32 staging buffer stays small for multi-GB pools.
    slab = max(1, (1 << 26) // (num_kv_heads * block_size * head_dim))
    for t in (k, v):
        for b0 in range(0, num_blocks, slab):
            b1 = min(num_blocks, b0 + slab)
            t[b0:b1] = torch.randn((b1 - b0,) + shape[1:], generator=gen, device=device,
                                   dtype=torch.float32).to(torch.bfloat16)
    if poison:
        poison_unused(k, v, block_table, lengths)
    return Workload(cfg=cfg, q=q, k_cache=k, v_cache=v,
                    block_table=torch.from_numpy(np.ascontiguousarray(block_table)).to(device),
                    seq_lens=torch.from_numpy(np.ascontiguousarray(lengths, dtype=np.int32)).to(device),
                    scale=1.0 / math.sqrt(head_dim))


def scatter_logical(k_logical: list, v_logical: list, num_kv_heads: int, block_size: int,
                    block_table: np.ndarray, num_blocks: int):
    """Place per-sequence logical K/V ([L_s, Hkv, d] each) into a paged pool
    through ``block_table``.  Returns (k_cache, v_cache) with unused slots NaN."""
    d = k_logical[0].shape[-1] if k_logical else HEAD_DIM
    dtype = k_logical[0].dtype if k_logical else torch.bfloat16
    k = torch.full((num_blocks, num_kv_heads, block_size, d), float("nan"), dtype=dtype)
    v = torch.full((num_blocks, num_kv_heads, block_size, d), float("nan"), dtype=dtype)
    for s, (ks, vs) in enumerate(zip(k_logical, v_logical)):
        L = ks.shape[0]
        for t in range(L):
            b = int(block_table[s, t // block_size])
            k[b, :, t % block_size, :] = ks[t]
            v[b, :, t % block_size, :] = vs[t]
    return k, v


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    """bf16 tensor -> numpy uint16 bit patterns (host copy)."""
    return t.detach().contiguous().cpu().view(torch.int16).numpy().view(np.uint16)


# --- chunked prefill -------------------------------------------------------
#
# A prefill batch: sequence s already holds `prior` cached tokens (earlier
# chunks of its prompt) and brings `new` prompt tokens whose K/V the serving
# engine has written into the cache; the new tokens are the queries.  The
# shapes follow the Llama-3-8B layer of the decode workloads; the chunk sizes
# are those of chunked-prefill serving (hundreds to a few thousand tokens).

@dataclass(frozen=True)
class PrefillConfig:
    key: str
    name: str
    num_seqs: int
    num_q_heads: int
    num_kv_heads: int
    block_size: int
    new_tokens: tuple    # (lo, hi) inclusive, uniform
    prior_tokens: tuple  # (lo, hi) inclusive, uniform
    seed: int
    head_dim: int = HEAD_DIM


PREFILL_CONFIGS = {
    "p1": PrefillConfig(key="p1", name="tiny-prefill-gqa4", num_seqs=3, num_q_heads=8, num_kv_heads=2,
                        block_size=16, new_tokens=(1, 300), prior_tokens=(0, 400), seed=10),
    "p2": PrefillConfig(key="p2", name="llama3-8b-chunked-prefill", num_seqs=8, num_q_heads=32, num_kv_heads=8,
                        block_size=16, new_tokens=(512, 2048), prior_tokens=(0, 4096), seed=11),
}


@dataclass
class PrefillWorkload:
    cfg: PrefillConfig | None
    q: torch.Tensor            # [T, Hq, d] bf16, the new tokens of all sequences
    k_cache: torch.Tensor      # [NB, Hkv, bs, d] bf16
    v_cache: torch.Tensor
    block_table: torch.Tensor  # [S, mbps] int32
    seq_lens: torch.Tensor     # [S] int32, prior + new
    q_start: torch.Tensor      # [S + 1] int32
    q_lens: np.ndarray         # [S] int32 (host copy)
    lengths: np.ndarray        # [S] int32 (host copy of seq_lens)
    scale: float

    @property
    def max_q_len(self) -> int:
        return int(self.q_lens.max(initial=0))

    def to(self, device) -> "PrefillWorkload":
        return PrefillWorkload(cfg=self.cfg, q=self.q.to(device), k_cache=self.k_cache.to(device),
                               v_cache=self.v_cache.to(device), block_table=self.block_table.to(device),
                               seq_lens=self.seq_lens.to(device), q_start=self.q_start.to(device),
                               q_lens=self.q_lens, lengths=self.lengths, scale=self.scale)


def make_prefill_workload(cfg: PrefillConfig | str, device="cpu", poison: bool = True,
                          new=None, prior=None, num_q_heads: int | None = None,
                          num_kv_heads: int | None = None, block_size: int | None = None,
                          spare_blocks: int = 0, seed: int | None = None) -> PrefillWorkload:
    """Build a prefill batch; `new` / `prior` override the sampled token
    counts and the head / block sizes can be overridden for edge cases."""
    if isinstance(cfg, str):
        cfg = PREFILL_CONFIGS[cfg]
    seed = cfg.seed if seed is None else seed
    Hq = num_q_heads or cfg.num_q_heads
    Hkv = num_kv_heads or cfg.num_kv_heads
    bs = block_size or cfg.block_size
    rng = np.random.default_rng(seed)
    if new is None:
        new = rng.integers(cfg.new_tokens[0], cfg.new_tokens[1], size=cfg.num_seqs, endpoint=True)
    if prior is None:
        prior = rng.integers(cfg.prior_tokens[0], cfg.prior_tokens[1], size=len(new), endpoint=True)
    q_lens = np.asarray(new, dtype=np.int32)
    lengths = (np.asarray(prior, dtype=np.int64) + q_lens).astype(np.int32)
    S = len(lengths)
    mbps = max(1, (int(lengths.max(initial=0)) + bs - 1) // bs)
    num_blocks = max(1, blocks_needed(lengths, bs) + spare_blocks)
    bt = build_block_table(lengths, bs, mbps, num_blocks, np.random.default_rng(seed + 1000))
    device = torch.device(device)
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed))
    T = int(q_lens.sum())
    q = torch.randn((T, Hq, cfg.head_dim), generator=gen, device=device, dtype=torch.float32).to(torch.bfloat16)
    shape = (num_blocks, Hkv, bs, cfg.head_dim)
    k = torch.empty(shape, device=device, dtype=torch.bfloat16)
    v = torch.empty(shape, device=device, dtype=torch.bfloat16)
    slab = max(1, (1 << 26) // (Hkv * bs * cfg.head_dim))
    for t in (k, v):
        for b0 in range(0, num_blocks, slab):
            b1 = min(num_blocks, b0 + slab)
            t[b0:b1] = torch.randn((b1 - b0,) + shape[1:], generator=gen, device=device,
                                   dtype=torch.float32).to(torch.bfloat16)
    if poison:
        poison_unused(k, v, bt, lengths)
    q_start = np.concatenate([[0], np.cumsum(q_lens)]).astype(np.int32)
    return PrefillWorkload(cfg=cfg, q=q, k_cache=k, v_cache=v,
                           block_table=torch.from_numpy(bt).to(device),
                           seq_lens=torch.from_numpy(np.ascontiguousarray(lengths)).to(device),
                           q_start=torch.from_numpy(q_start).to(device), q_lens=q_lens, lengths=lengths,
                           scale=1.0 / math.sqrt(cfg.head_dim))
