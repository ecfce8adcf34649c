#!/usr/bin/env python
"""Benchmark of paged GQA decode attention on GB300.

One step = one decode-attention call (one kernel: the split-KV streaming
pass with the log-sum-exp merge of cut pieces fused in) over one batch of a
named synthetic workload whose inputs are already resident in HBM.  L2 is
flushed before every timed step, outside the timed interval (a 2x-L2 buffer
written and read back, so that no dirty lines are written back inside the
next step), and each step is timed with CUDA events on the launching
stream.

Prints one JSON line.  By default the four large workloads run one after
another in this process, each timed for --steps steps: the headline
(value, roofline, e2e, cpu_baseline, clocks) is the largest single-GPU
workload, the 70B-shaped 256-sequence batch (block 32, contexts
U[2048, 8192] in a 6 GiB pool); the Llama-3-8B, long-thinking and
mixed-phase batches follow under "per_config", each with its own roofline
fraction, e2e figure and clock record.  --config k times workload k alone.
--impl reference times the fp64 CPU oracle on the host cores instead
(bounded samples of the same workload).

Multi-GPU (torchrun, one process per GPU): every rank runs its own batch of
the workload (weak scaling, no collective on the data path); the value is
the KV bytes of all ranks over the slowest rank's time.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "decode-attention KV-read GB/s & fraction of HBM peak; decode tokens/s (1 GB300)"
FALLBACK_HBM_GBS = 6800.0
NOMINAL_HBM_GBS = 7900.0  # NVIDIA's GB300 HBM3e figure, for a labelled second fraction only
# Layers of the model each workload is shaped after (8B: 32, 32B: 64, 70B: 80).
MODEL_LAYERS = {1: None, 2: 32, 3: 32, 4: 64, 5: 80}
PROFILES = os.path.join(ROOT, "profiles")
HEADLINE_CONFIG = 5            # the largest workload that fits one GPU
DEFAULT_CONFIGS = (5, 2, 3, 4)  # headline first, then the other large workloads
PREFILL_SUMMARY = os.path.join(ROOT, "profiles", "ps_prefill_kernel_llama3-8b-chunked-prefill.md")
PREFILL_SOURCE = os.path.join(ROOT, "paper_2608_21719_gb300", "csrc", "ps_prefill.cu")
FALLBACK_BF16_TFLOPS = 1900.0
KERNEL_SOURCE = os.path.join(ROOT, "paper_2608_21719_gb300", "csrc", "ps_decode_kernels.cu")
CLOCK_QUERY = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
               "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
               "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")


def parse_args(argv=None):
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", type=int, default=None, choices=[1, 2, 3, 4, 5],
                    help="time this workload alone (default: workloads 5, 2, 3, 4, headline 5)")
    ap.add_argument("--cpu-seconds", type=float, default=12.0,
                    help="CPU time budget of the oracle baseline sample")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--prefill", action="store_true",
                    help="time the tcgen05 chunked-prefill attention on the 8-sequence Llama-3-8B "
                         "prefill batch instead (metric: TFLOP/s)")
    ap.add_argument("--transfer", choices=["pack", "unpack"], default=None,
                    help="time the KV hand-off gather (pack) or scatter (unpack) of the whole batch instead")
    ap.add_argument("--min-stages", type=int, default=0,
                    help="smallest share of one worker warp, in 16-token tiles (0: library default)")
    ap.add_argument("--sms", type=int, default=0,
                    help="size the persistent grid for this many SMs (0: all); a proxy for lower SM throughput")
    ap.add_argument("--append", action="store_true",
                    help="time the fused step: append the current token's K/V to the cache, then attend")
    ap.add_argument("--flush", choices=["write-read", "write"], default="write-read",
                    help="L2 flush between steps: write a 2x-L2 buffer, then read it back so that "
                         "L2 holds clean lines (default), or only write it (leaves dirty lines whose "
                         "write-back lands inside the next timed step)")
    return ap.parse_args(argv)


# ----------------------------------------------------------------- helpers --

def dist_env():
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("LOCAL_RANK", "0")),
            int(os.environ.get("WORLD_SIZE", "1")))


def slowest_rank_ms(total_ms: float, device) -> float:
    """Max over ranks of the timed region (the whole-job time); identity
    without an initialised process group."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(total_ms)
    t = torch.tensor([float(total_ms)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(bytes_per_step: int, steps: int, world: int, slowest_ms: float) -> float:
    """Whole-job GB/s: every rank moved bytes_per_step per step (weak scaling)."""
    return bytes_per_step * steps * world / (slowest_ms * 1e-3) / 1e9


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def decode_profile_summary(workload: str) -> str:
    """Path of the committed ncu summary of the decode kernel on a workload."""
    return os.path.join(PROFILES, "ps_decode_kernel_%s.md" % workload)


def profiled_traffic(summary, source=KERNEL_SOURCE, workload=None):
    """Per-launch DRAM bytes (dram__bytes_read.sum + dram__bytes_write.sum)
    of a kernel from its committed ncu summary of this workload, or None
    when there is no summary for it, it names another workload, or the
    kernel source changed since the counters were taken."""
    try:
        text = open(summary).read()
        src_hash = hashlib.sha256(open(source, "rb").read()).hexdigest()
    except OSError:
        return None
    vals = {}
    for line in text.splitlines():
        line = line.strip().lstrip("-* ")
        if ":" in line:
            k, v = line.split(":", 1)
            vals[k.strip().strip("`")] = v.strip().strip("`")
    if vals.get("kernel_source_sha256") != src_hash:
        return None
    if workload is not None and vals.get("workload") != workload:
        return None
    try:
        return int(float(vals["traffic_bytes_per_launch"]))
    except (KeyError, ValueError):
        return None


class ClockSampler:
    """nvidia-smi sampling (read-only queries) of SM clocks and throttle
    reasons, polled every 5 ms.  mark_start()/mark_end() bracket the timed
    region on the host clock; the summary counts the samples whose
    nvidia-smi timestamps fall inside it (falling back to all samples taken
    while the sampler ran when the region is shorter than one poll)."""

    POLL_MS = 5

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None
        self.t0 = self.t1 = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(prefix="ps_clocks_", suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + CLOCK_QUERY, "--format=csv,noheader,nounits",
                 "-lms", str(self.POLL_MS)], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None
        time.sleep(0.3)
        return self

    def mark_start(self):
        self.t0 = time.time()

    def mark_end(self):
        self.t1 = time.time()

    def __exit__(self, *exc):
        time.sleep(0.05)
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    @staticmethod
    def _stamp(text):
        import datetime
        for fmt in ("%Y/%m/%d %H:%M:%S.%f", "%Y/%m/%d %H:%M:%S"):
            try:
                return datetime.datetime.strptime(text.strip(), fmt).timestamp()
            except ValueError:
                continue
        return None

    def summary(self):
        if self.proc is None or self.path is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        rows = []
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) >= 10:
                rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}

        def num(x):
            try:
                return float(x)
            except ValueError:
                return None
        inside = rows
        if self.t0 is not None and self.t1 is not None:
            # nvidia-smi prints local wall-clock time; allow one poll of slack at each end.
            slack = self.POLL_MS * 1e-3
            sel = [r for r in rows if (lambda t: t is not None and self.t0 - slack <= t <= self.t1 + slack)(
                self._stamp(r[0]))]
            if sel:
                inside = sel
        sm = [num(r[2]) for r in inside if num(r[2]) is not None]
        mx = [num(r[3]) for r in inside if num(r[3]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in inside for i in range(4) if r[6 + i].lower() == "active"})
        power = [num(r[4]) for r in inside if num(r[4]) is not None]
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(inside), "samples_total": len(rows),
                "in_region": inside is not rows, "poll_ms": self.POLL_MS,
                "region_ms": None if self.t0 is None or self.t1 is None else round((self.t1 - self.t0) * 1e3, 2),
                "power_w_max": max(power) if power else None}


def sample_for_oracle(wl, seq_idx, token_cap=None):
    """Host copy of sequences ``seq_idx`` (optionally only their first
    ``token_cap`` tokens) as a compact paged workload for the oracle."""
    import numpy as np
    import torch
    from paper_2608_21719_gb300 import inputs
    bs = wl.block_size
    lens = wl.seq_lens[seq_idx].cpu().numpy().astype(np.int64)
    if token_cap is not None:
        lens = np.minimum(lens, token_cap)
    bt = wl.block_table[seq_idx].cpu().numpy()
    pages = [bt[i, :(int(L) + bs - 1) // bs] for i, L in enumerate(lens)]
    flat = torch.from_numpy(np.concatenate(pages).astype(np.int64)).to(wl.k_cache.device)
    k = wl.k_cache.index_select(0, flat).cpu()
    v = wl.v_cache.index_select(0, flat).cpu()
    nbt = np.full((len(seq_idx), max(1, max(len(p) for p in pages))), -1, dtype=np.int32)
    pos = 0
    for i, p in enumerate(pages):
        nbt[i, :len(p)] = np.arange(pos, pos + len(p))
        pos += len(p)
    return inputs.Workload(cfg=None, q=wl.q[seq_idx].cpu(), k_cache=k, v_cache=v,
                           block_table=torch.from_numpy(nbt), seq_lens=torch.from_numpy(lens.astype(np.int32)),
                           scale=wl.scale)


def time_oracle(sub, threads):
    import oracle
    from paper_2608_21719_gb300 import inputs, roofline
    args = (inputs.bf16_bits(sub.q), inputs.bf16_bits(sub.k_cache), inputs.bf16_bits(sub.v_cache),
            sub.block_table.numpy(), sub.seq_lens.numpy(), sub.num_kv_heads, sub.scale)
    t0 = time.perf_counter()
    oracle.decode_attention(*args, num_threads=threads)
    dt = time.perf_counter() - t0
    kv = roofline.algorithmic_bytes(sub.seq_lens.numpy(), sub.num_q_heads, sub.num_kv_heads, sub.head_dim,
                                    sub.block_size)["kv"]
    return dt, kv


def choose_oracle_sample(wl, budget_s, threads):
    """Sequences (in a fixed seeded order) and a token cap sized so that one
    oracle run over them takes about ``budget_s`` seconds."""
    import numpy as np
    order = list(np.random.default_rng(12345).permutation(wl.num_seqs))
    probe = sample_for_oracle(wl, order[:1], token_cap=512)
    dt, kv = time_oracle(probe, threads)
    rate = kv / max(dt, 1e-6)  # KV bytes per second of the oracle
    want = rate * budget_s
    lens = wl.seq_lens.cpu().numpy()
    per_tok = 2 * wl.num_kv_heads * wl.head_dim * 2
    chosen, acc = [], 0
    for s in order:
        b = int(lens[s]) * per_tok
        if acc + b > want and chosen:
            break
        chosen.append(int(s))
        acc += b
    cap = None
    if len(chosen) == 1 and acc > want:
        cap = max(16, int(want // per_tok))
    return chosen, cap


# ------------------------------------------------------------- our arm ------

def workload_config(cfg, wl, alg, flush_mb, world, append=False):
    """The "config" object of a bench line; both arms print the same one for
    the same workload."""
    lens = wl.seq_lens.cpu().numpy()
    return {
        "workload": cfg.name,
        "num_seqs": wl.num_seqs, "num_q_heads": wl.num_q_heads, "num_kv_heads": wl.num_kv_heads,
        "head_dim": wl.head_dim, "block_size": wl.block_size, "lengths": list(cfg.lengths),
        "seed": cfg.seed, "total_tokens": int(lens.sum()), "kv_bytes": alg["kv"],
        "pool_blocks": wl.num_blocks,
        "l2": "flushed before every step, outside the timed interval: write then read of a %d MB buffer" % flush_mb,
        "parallelism": "replicas" if world == 1 else "dp%d (independent batches per GPU)" % world,
        "step": "append current token K/V + attend" if append else "attend",
    }


def flush_bytes(dev) -> int:
    import torch
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    return max(2 * l2, 64 << 20) // 4 * 4


def gpu_index_of(local_rank: int) -> str:
    visible = [x.strip() for x in os.environ.get("CUDA_VISIBLE_DEVICES", "").split(",") if x.strip()]
    return visible[local_rank] if local_rank < len(visible) else str(local_rank)


def measure_decode(args, key, dev, rank, local_rank, world):
    """Time one workload: kernel-only steps (CUDA events on the launching
    stream, L2 flushed before each), then the end-to-end loop through the
    public API with host buffers.  Returns (fields of the JSON line, the
    workload, its algorithmic bytes) on every rank."""
    import torch
    import torch.distributed as dist

    from paper_2608_21719_gb300 import inputs, ps_decode, roofline

    cfg = inputs.CONFIGS[key]
    wl = inputs.make_workload(cfg, device=dev, poison=False)
    lens = wl.seq_lens.cpu().numpy()
    alg = roofline.algorithmic_bytes(lens, wl.num_q_heads, wl.num_kv_heads, wl.head_dim, wl.block_size)

    attn = ps_decode.DecodeAttention.for_workload(wl, num_sms=args.sms, min_stages_per_worker=args.min_stages)
    out = torch.empty_like(wl.q)
    stream = torch.cuda.current_stream(dev)
    flush_buf = torch.empty(flush_bytes(dev) // 4, dtype=torch.int32, device=dev)
    flush_sink = torch.empty((), dtype=torch.int32, device=dev)

    def flush():
        """Evict the inputs from L2 between steps, outside the timed interval."""
        flush_buf.zero_()
        if args.flush == "write-read":
            torch.amax(flush_buf, dim=0, out=flush_sink)

    if args.append:
        gen = torch.Generator(device=dev)
        gen.manual_seed(cfg.seed + 77)
        k_new = torch.randn((wl.num_seqs, wl.num_kv_heads, wl.head_dim), generator=gen, device=dev).to(torch.bfloat16)
        v_new = torch.randn((wl.num_seqs, wl.num_kv_heads, wl.head_dim), generator=gen, device=dev).to(torch.bfloat16)

    def step():
        if args.append:
            attn.append(wl.q, k_new, v_new, wl.k_cache, wl.v_cache, wl.block_table, wl.seq_lens, out=out,
                        scale=wl.scale, stream=stream)
        else:
            attn(wl.q, wl.k_cache, wl.v_cache, wl.block_table, wl.seq_lens, out=out, scale=wl.scale, stream=stream)

    for _ in range(max(args.warmup, 3)):
        flush()
        step()
    torch.cuda.synchronize(dev)
    assert attn.device_status() == 0, "device status flags raised during warm-up"

    K = args.steps
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(K)]
    for e in ev:
        for x in e:
            x.record(stream)  # create the CUDA events before the timed region
    n_launch0 = ps_decode.ps_decode_launch_count()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    with ClockSampler(gpu_index_of(local_rank)) as clk:
        clk.mark_start()
        for k in range(K):
            flush()
            ps_decode.ps_decode_plan_set_timing_events(attn.plan, *ev[k])
            step()
        torch.cuda.synchronize(dev)
        clk.mark_end()
    if world > 1:
        dist.barrier()
    launches = ps_decode.ps_decode_launch_count() - n_launch0
    ps_decode.ps_decode_plan_set_timing_events(attn.plan, None, None)
    assert attn.device_status() == 0, "device status flags raised during the timed steps"
    step_ms = [e[0].elapsed_time(e[1]) for e in ev]
    total_ms = slowest_rank_ms(sum(step_ms), dev)

    # End to end through the public API with host buffers: per step, copy the
    # step's inputs (queries, block table, lengths) from pinned host memory,
    # run the call, and read the output back.  The KV cache is the serving
    # engine's resident state and stays in HBM.
    # The three inputs travel as one packed pinned buffer (one copy per step)
    # into one device buffer that the call reads through three pointers.  As a
    # serving loop would, the copies of step i+1 and the read-back of step i-1
    # overlap the call of step i: two buffer sets, host-to-device copies,
    # calls and read-backs on three streams ordered by events; the time is
    # the whole loop's.  Every step still moves its own inputs in and its
    # output out.  No L2 flush in between: each step reads the whole K/V pool,
    # which is larger than L2.
    packs = [packed_inputs([wl.q, wl.block_table, wl.seq_lens], dev) for _ in range(2)]
    outs = [torch.empty_like(out) for _ in range(2)]
    outs_h = [torch.empty(out.shape, dtype=out.dtype).pin_memory() for _ in range(2)]
    h2d_s, d2h_s = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    ev_in = [torch.cuda.Event() for _ in range(2)]
    ev_k = [torch.cuda.Event() for _ in range(2)]
    ev_out = [torch.cuda.Event() for _ in range(2)]
    e2e_steps = max(10, min(K, 200))

    def e2e_loop(nsteps):
        for i in range(nsteps):
            b = i % 2
            (_, stage_h, (q_d, bt_d, sl_d), stage_d) = packs[b]
            with torch.cuda.stream(h2d_s):
                if i >= 2:
                    h2d_s.wait_event(ev_k[b])  # step i-2 has finished reading buffer set b
                stage_d.copy_(stage_h, non_blocking=True)
                ev_in[b].record(h2d_s)
            stream.wait_event(ev_in[b])
            if i >= 2:
                stream.wait_event(ev_out[b])  # step i-2's output has been read back
            attn(q_d, wl.k_cache, wl.v_cache, bt_d, sl_d, out=outs[b], scale=wl.scale, stream=stream)
            ev_k[b].record(stream)
            with torch.cuda.stream(d2h_s):
                d2h_s.wait_event(ev_k[b])
                outs_h[b].copy_(outs[b], non_blocking=True)
                ev_out[b].record(d2h_s)

    e2e_loop(4)
    torch.cuda.synchronize(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(h2d_s)
    e2e_loop(e2e_steps)
    d2h_s.wait_event(ev_out[(e2e_steps - 1) % 2])
    e1.record(d2h_s)
    torch.cuda.synchronize(dev)
    e2e_ms = e0.elapsed_time(e1) / e2e_steps
    h2d = packs[0][1].numel()
    d2h = outs_h[0].numel() * 2
    assert torch.equal(outs_h[(e2e_steps - 1) % 2], outs[(e2e_steps - 1) % 2].cpu())
    # Whole job: every rank's bytes over the slowest rank's loop.
    e2e_total_ms = slowest_rank_ms(e2e_ms * e2e_steps, dev)
    e2e_value = job_throughput(alg["kv"], e2e_steps, world, e2e_total_ms)
    info = attn.info()
    attn.close()
    del packs, outs, outs_h, flush_buf

    hbm_peak, peak_kind = measured_peaks()
    ms_per_step = total_ms / K
    value = job_throughput(alg["kv"], K, world, total_ms)
    achieved = alg["total"] / (ms_per_step * 1e-3) / 1e9
    layers = MODEL_LAYERS.get(key)
    fields = {
        "value": round(value, 2),
        "ms_per_step": round(ms_per_step, 5),
        "config": workload_config(cfg, wl, alg, flush_bytes(dev) >> 20, world, args.append),
        "frac_of_hbm_peak": round(achieved / hbm_peak, 4),
        "decode_tokens_per_s": round(wl.num_seqs * world * K / (total_ms * 1e-3), 1),
        # Context only: one attention call per layer, so a whole model's
        # decode step over this batch needs n_layers of them.
        "attention_only_tokens_per_s": (
            None if layers is None else
            {"n_layers": layers, "value": round(wl.num_seqs * world * K / (total_ms * 1e-3) / layers, 1)}),
        "kernel_ms": {"mean": round(ms_per_step, 5), "median": round(statistics.median(step_ms), 5),
                      "min": round(min(step_ms), 5), "max": round(max(step_ms), 5)},
        "frac_of_nominal_hbm": round(achieved / NOMINAL_HBM_GBS, 4),
        "roofline": {
            "kernel": "ps_decode_kernel",
            "bound": "hbm",
            "achieved": round(achieved, 1),
            "peak": hbm_peak,
            "peak_kind": peak_kind + " (copy bandwidth, burst)",
            "unit": "GB/s",
            "frac": round(achieved / hbm_peak, 4),
            "traffic": None if (args.sms or args.min_stages or args.append) else profiled_traffic(
                decode_profile_summary(cfg.name), workload=cfg.name),
            "algorithmic_bytes_per_launch": alg["total"],
        },
        "e2e": {"value": round(e2e_value, 2), "unit": "GB/s",
                "ms_per_step": round(e2e_total_ms / e2e_steps, 5), "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "steps": e2e_steps,
                "overlap": "copies of step i+1 and read-back of step i-1 overlap the call of step i "
                           "(two buffer sets, three streams); time = whole loop / steps",
                "l2": "not flushed: each step reads the whole K/V pool, larger than L2"},
        "gpu_launches": int(launches),
        "clocks": clk.summary(),
        "plan": info,
    }
    return fields, wl, alg


def cpu_baseline_for(wl, budget_s):
    """The oracle, as it stands, on the host cores over a bounded sample of
    the workload (whole sequences in a seeded order, about budget_s of CPU
    time per run, repeated to about budget_s in total)."""
    threads = os.cpu_count() or 1
    chosen, cap = choose_oracle_sample(wl, budget_s, threads)
    sub = sample_for_oracle(wl, chosen, token_cap=cap)
    spent, kv, reps = 0.0, 0, 0
    while reps == 0 or spent < 0.8 * budget_s:
        dt, b = time_oracle(sub, threads)
        spent += dt
        kv += b
        reps += 1
    return {
        "value": round(kv / spent / 1e9, 4), "unit": "GB/s", "cores": threads, "kind": "oracle",
        "sample": "%d of %d sequences%s of this workload x %d runs, fp64 oracle, %.1f s" % (
            len(chosen), wl.num_seqs, "" if cap is None else " (first %d tokens)" % cap, reps, spent),
    }


def run_ours(args):
    import torch
    import torch.distributed as dist

    rank, local_rank, world = dist_env()
    if world > 1 and not dist.is_initialized():
        dist.init_process_group("nccl")
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    keys = (args.config,) if args.config is not None else DEFAULT_CONFIGS
    results = {}
    head_wl = None
    for key in keys:
        fields, wl, _ = measure_decode(args, key, dev, rank, local_rank, world)
        results[key] = fields
        if key == keys[0] and rank == 0 and not args.no_cpu_baseline:
            results[key]["cpu_baseline"] = cpu_baseline_for(wl, args.cpu_seconds)
        del wl
        torch.cuda.empty_cache()
    if world > 1:
        dist.barrier()
    if rank != 0:
        return None
    head = results[keys[0]]
    line = {
        "metric": METRIC,
        "value": head["value"],
        "unit": "GB/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": head["ms_per_step"],
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic",
    }
    line.update(head)
    if len(keys) > 1:
        line["per_config"] = {
            results[k]["config"]["workload"]: {
                "value": results[k]["value"], "unit": "GB/s", "ms_per_step": results[k]["ms_per_step"],
                "decode_tokens_per_s": results[k]["decode_tokens_per_s"],
                "roofline": {x: results[k]["roofline"][x] for x in ("achieved", "peak", "frac", "traffic",
                                                                     "algorithmic_bytes_per_launch")},
                "e2e": {x: results[k]["e2e"][x] for x in ("value", "unit", "ms_per_step", "h2d_bytes_per_step",
                                                          "d2h_bytes_per_step")},
                "kernel_ms": results[k]["kernel_ms"],
                "gpu_launches": results[k]["gpu_launches"],
                "clocks": results[k]["clocks"],
                "config": results[k]["config"],
            } for k in keys[1:]}
        line["gpu_launches"] = sum(results[k]["gpu_launches"] for k in keys)
        line["gpu_launches_note"] = "headline workload %d; all timed regions of this run: %d" % (
            head["gpu_launches"], line["gpu_launches"])
    return line


# ------------------------------------------------------- KV hand-off ------

def run_transfer(args):
    """Pack (or unpack) every sequence of the workload between its paged pool
    and contiguous per-sequence buffers; metric: bytes read + written / time."""
    import numpy as np
    import torch

    from paper_2608_21719_gb300 import inputs, ps_decode

    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    cfg = inputs.CONFIGS[args.config if args.config is not None else HEADLINE_CONFIG]
    wl = inputs.make_workload(cfg, device=dev, poison=False)
    lens = wl.seq_lens.cpu().numpy().astype(np.int64)
    Hkv, d, bs = wl.num_kv_heads, wl.head_dim, wl.block_size
    sizes = 2 * Hkv * lens * d
    off = torch.from_numpy(np.concatenate([[0], np.cumsum(sizes)[:-1]]).astype(np.int64)).to(dev)
    buf = torch.empty(int(sizes.sum()), dtype=torch.bfloat16, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream(dev)
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    flush_buf = torch.empty(max(2 * l2, 64 << 20) // 4, dtype=torch.int32, device=dev)
    sink = torch.empty((), dtype=torch.int32, device=dev)
    args_common = (wl.block_table, wl.max_blocks_per_seq, wl.seq_lens, wl.num_seqs, Hkv, d, bs, wl.num_blocks)

    def step():
        if args.transfer == "pack":
            ps_decode.ps_kv_pack(wl.k_cache, wl.v_cache, *args_common, off, buf, status, stream)
        else:
            ps_decode.ps_kv_unpack(buf, off, *args_common, wl.k_cache, wl.v_cache, status, stream)

    for _ in range(max(args.warmup, 3)):
        flush_buf.zero_(); torch.amax(flush_buf, dim=0, out=sink)
        step()
    torch.cuda.synchronize(dev)
    K = args.steps
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    launches0 = ps_decode.ps_decode_launch_count()
    with ClockSampler(gpu_index_of(0)) as clk:
        clk.mark_start()
        for a, b in ev:
            flush_buf.zero_(); torch.amax(flush_buf, dim=0, out=sink)
            a.record(stream)
            step()
            b.record(stream)
        torch.cuda.synchronize(dev)
        clk.mark_end()
    launches = ps_decode.ps_decode_launch_count() - launches0
    assert int(status.item()) == 0
    ms = statistics.mean(a.elapsed_time(b) for a, b in ev)
    moved = 2 * int(sizes.sum()) * 2  # every element read once and written once
    peak, kind = measured_peaks()
    gbs = moved / (ms * 1e-3) / 1e9
    return {
        "metric": "KV hand-off %s GB/s (read + write)" % args.transfer, "value": round(gbs, 2), "unit": "GB/s",
        "n_gpus": 1, "steps": K, "warmup": args.warmup, "ms_per_step": round(ms, 5), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": cfg.name, "bytes_moved": moved, "l2": "write-then-read flush before every step"},
        "roofline": {"kernel": "ps_kv_transfer_kernel", "bound": "hbm", "achieved": round(gbs, 1), "peak": peak,
                     "peak_kind": kind + " (copy bandwidth)", "unit": "GB/s", "frac": round(gbs / peak, 4),
                     "traffic": None},
        "gpu_launches": launches,
        "clocks": clk.summary(),
    }


def bf16_peak():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["bf16_tflops"]), "measured"
    except Exception:
        return FALLBACK_BF16_TFLOPS, "fallback"


def time_prefill_oracle(wl, budget_s, threads):
    """The prefill oracle on a causal prefix of one sequence's chunk (the
    first n new tokens, which later tokens cannot influence), n grown until
    one call takes about budget_s.  Returns (flops/s, description)."""
    import numpy as np

    import oracle
    from paper_2608_21719_gb300 import inputs, roofline

    s = int(np.argmax(wl.q_lens))
    Q, L = int(wl.q_lens[s]), int(wl.lengths[s])
    prior = L - Q
    bt = wl.block_table[s:s + 1].cpu().numpy()
    k_bits = inputs.bf16_bits(wl.k_cache)
    v_bits = inputs.bf16_bits(wl.v_cache)
    q0 = int(wl.q_start[s].item())
    Hkv = wl.k_cache.shape[1]
    n = 4
    while True:
        q_bits = inputs.bf16_bits(wl.q[q0:q0 + n])
        t0 = time.perf_counter()
        oracle.prefill_attention(q_bits, k_bits, v_bits, bt, np.asarray([prior + n], dtype=np.int32),
                                 np.asarray([0, n], dtype=np.int32), Hkv, wl.scale, num_threads=threads)
        dt = time.perf_counter() - t0
        fl = roofline.prefill_flops([prior + n], [n], wl.q.shape[1], wl.q.shape[2])
        if dt >= budget_s or n >= Q:
            return fl / dt, "sequence %d: first %d of its %d new tokens over %d cached (%.2f GFLOP)" % (
                s, n, Q, prior, fl / 1e9)
        n = min(Q, max(n + 1, int(n * min(8.0, 1.3 * budget_s / max(dt, 1e-4)))))


def run_prefill(args):
    """Chunked-prefill attention (tcgen05) over the whole 8-sequence batch;
    metric: causal attention FLOPs / time."""
    import torch

    from paper_2608_21719_gb300 import inputs, ps_decode, roofline

    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    cfg = inputs.PREFILL_CONFIGS["p2"]
    wl = inputs.make_prefill_workload(cfg, device=dev)
    Hq, d = wl.q.shape[1], wl.q.shape[2]
    flops = roofline.prefill_flops(wl.lengths, wl.q_lens, Hq, d)
    out = torch.empty_like(wl.q)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream(dev)
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    flush_buf = torch.empty(max(2 * l2, 64 << 20) // 4, dtype=torch.int32, device=dev)
    sink = torch.empty((), dtype=torch.int32, device=dev)

    def step():
        ps_decode.prefill_attention(wl.q, wl.k_cache, wl.v_cache, wl.block_table, wl.seq_lens, wl.q_start,
                                    wl.max_q_len, out=out, scale=wl.scale, device_status=status,
                                    stream=stream.cuda_stream)

    def flush():
        flush_buf.zero_()
        torch.amax(flush_buf, dim=0, out=sink)

    for _ in range(max(args.warmup, 3)):
        flush()
        step()
    torch.cuda.synchronize(dev)
    K = args.steps
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    launches0 = ps_decode.ps_decode_launch_count()
    with ClockSampler(gpu_index_of(0)) as clk:
        clk.mark_start()
        for a, b in ev:
            flush()
            a.record(stream)
            step()
            b.record(stream)
        torch.cuda.synchronize(dev)
        clk.mark_end()
    launches = ps_decode.ps_decode_launch_count() - launches0
    assert int(status.item()) == 0, "device status %d" % int(status.item())
    ms = statistics.mean(a.elapsed_time(b) for a, b in ev)
    tflops = flops / (ms * 1e-3) / 1e12

    # End to end: pinned host Q and metadata in, output back, every step, with
    # the copies of step i+1 and the read-back of step i-1 overlapping the call
    # of step i (two buffer sets, three streams); time = whole loop / steps.
    packs = [packed_inputs([wl.q, wl.block_table, wl.seq_lens, wl.q_start], dev) for _ in range(2)]
    outs = [torch.empty_like(out) for _ in range(2)]
    outs_h = [torch.empty(out.shape, dtype=out.dtype, pin_memory=True) for _ in range(2)]
    h2d_s, d2h_s = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    ev_in = [torch.cuda.Event() for _ in range(2)]
    ev_k = [torch.cuda.Event() for _ in range(2)]
    ev_out = [torch.cuda.Event() for _ in range(2)]
    K2 = max(4, min(K, 50))

    def e2e_loop(nsteps):
        for i in range(nsteps):
            b = i % 2
            (_, stage_h, (q_d, bt_d, sl_d, qs_d), stage_d) = packs[b]
            with torch.cuda.stream(h2d_s):
                if i >= 2:
                    h2d_s.wait_event(ev_k[b])
                stage_d.copy_(stage_h, non_blocking=True)
                ev_in[b].record(h2d_s)
            stream.wait_event(ev_in[b])
            if i >= 2:
                stream.wait_event(ev_out[b])
            ps_decode.prefill_attention(q_d, wl.k_cache, wl.v_cache, bt_d, sl_d, qs_d, wl.max_q_len, out=outs[b],
                                        scale=wl.scale, device_status=status, stream=stream.cuda_stream)
            ev_k[b].record(stream)
            with torch.cuda.stream(d2h_s):
                d2h_s.wait_event(ev_k[b])
                outs_h[b].copy_(outs[b], non_blocking=True)
                ev_out[b].record(d2h_s)

    e2e_loop(2)
    torch.cuda.synchronize(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(h2d_s)
    e2e_loop(K2)
    d2h_s.wait_event(ev_out[(K2 - 1) % 2])
    e1.record(d2h_s)
    torch.cuda.synchronize(dev)
    e2e_ms = e0.elapsed_time(e1) / K2
    h2d = packs[0][1].numel()
    d2h = outs_h[0].numel() * 2

    peak, kind = bf16_peak()
    line = {
        "metric": "chunked-prefill attention TFLOP/s (causal, paged KV, tcgen05)", "value": round(tflops, 2),
        "unit": "TFLOP/s", "n_gpus": 1, "steps": K, "warmup": args.warmup, "ms_per_step": round(ms, 5),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": cfg.name, "num_seqs": cfg.num_seqs, "num_q_heads": Hq,
                   "num_kv_heads": wl.k_cache.shape[1], "head_dim": d, "block_size": wl.k_cache.shape[2],
                   "new_tokens": int(wl.q_lens.sum()), "cached_tokens": int(wl.lengths.sum()),
                   "flops_per_step": flops, "l2": "write-then-read flush before every step"},
        "roofline": {"kernel": "ps_prefill_kernel", "bound": "tensor", "achieved": round(tflops, 1), "peak": peak,
                     "peak_kind": kind + " (cuBLAS bf16 burst)", "unit": "TFLOP/s", "frac": round(tflops / peak, 4),
                     "traffic": profiled_traffic(PREFILL_SUMMARY, PREFILL_SOURCE)},
        "e2e": {"value": round(flops / (e2e_ms * 1e-3) / 1e12, 2), "unit": "TFLOP/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "steps": K2,
                "overlap": "copies of step i+1 and read-back of step i-1 overlap the call of step i "
                           "(two buffer sets, three streams); time = whole loop / steps"},
        "gpu_launches": launches,
        "clocks": clk.summary(),
    }
    if not args.no_cpu_baseline:
        threads = os.cpu_count() or 1
        rate, sample = time_prefill_oracle(wl, min(args.cpu_seconds, 20.0), threads)
        line["cpu_baseline"] = {"value": round(rate / 1e12, 6), "unit": "TFLOP/s", "cores": threads,
                                "kind": "oracle", "sample": sample}
    return line


def packed_inputs(tensors, dev, align=256):
    """One pinned host buffer and one device buffer holding copies of
    `tensors` at `align`-byte offsets; returns (host views, host buffer,
    device views, device buffer)."""
    import torch
    offs, total = [], 0
    for t in tensors:
        offs.append(total)
        total += (t.numel() * t.element_size() + align - 1) // align * align
    stage_h = torch.empty(max(total, align), dtype=torch.uint8).pin_memory()
    stage_d = torch.empty(max(total, align), dtype=torch.uint8, device=dev)

    def views(buf):
        return [buf[o:o + t.numel() * t.element_size()].view(t.dtype).view(t.shape) for o, t in zip(offs, tensors)]
    hv = views(stage_h)
    for h, t in zip(hv, tensors):
        h.copy_(t.cpu())
    return hv, stage_h, views(stage_d), stage_d


# ------------------------------------------------------- reference arm ------

def run_reference(args):
    """The oracle, as it stands, on the host cores: each step runs it over a
    bounded sample of the workload sized so that the whole run stays within
    a few minutes.  Same workload, metric and config object as our arm's
    headline."""
    import torch

    from paper_2608_21719_gb300 import inputs, roofline

    rank, _, world = dist_env()
    if rank != 0:
        return None
    key = args.config if args.config is not None else HEADLINE_CONFIG
    cfg = inputs.CONFIGS[key]
    if not torch.cuda.is_available() and key != 1:
        return {"impl": "reference", "unavailable": "workload %d needs a GPU to generate its inputs" % key}
    dev = torch.device("cuda", 0) if torch.cuda.is_available() else torch.device("cpu")
    wl = inputs.make_workload(cfg, device=dev, poison=False)
    alg = roofline.algorithmic_bytes(wl.seq_lens.cpu().numpy(), wl.num_q_heads, wl.num_kv_heads, wl.head_dim,
                                     wl.block_size)
    flush_mb = (flush_bytes(dev) >> 20) if dev.type == "cuda" else 0
    config = workload_config(cfg, wl, alg, flush_mb, world, args.append)
    threads = os.cpu_count() or 1
    budget = max(0.05, 150.0 / max(1, args.steps + args.warmup))
    chosen, cap = choose_oracle_sample(wl, budget, threads)
    sub = sample_for_oracle(wl, chosen, token_cap=cap)
    del wl
    for _ in range(args.warmup):
        time_oracle(sub, threads)
    t = 0.0
    kv = 0
    for _ in range(args.steps):
        dt, b = time_oracle(sub, threads)
        t += dt
        kv += b
    value = kv / t / 1e9
    sample = "%d of %d sequences%s per step" % (len(chosen), cfg.num_seqs,
                                                "" if cap is None else " (first %d tokens)" % cap)
    return {
        "impl": "reference",
        "metric": METRIC, "value": round(value, 4), "unit": "GB/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(t / args.steps * 1e3, 3), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": config,
        "cpu_baseline": {"value": round(value, 4), "unit": "GB/s", "cores": threads, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": round(value, 4), "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def main(argv=None):
    args = parse_args(argv)
    if args.impl == "reference":
        line = run_reference(args)
    elif args.prefill:
        line = run_prefill(args)
    elif args.transfer:
        line = run_transfer(args)
    else:
        line = run_ours(args)
    if line is not None:
        print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
