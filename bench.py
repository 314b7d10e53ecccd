#!/usr/bin/env python3
"""Decode-step benchmark of refusal-gated decoding on GB300.

One step = one pass of the whole hot path over one batch of the Llama-3-8B-shaped
workload (16 prompts x (1 greedy probe + 4 high-temperature sample rows), prompts
U[512, 2048] tokens, suffixes U[0, 256], 32 q / 8 kv heads, head dim 128, bf16 KV
in 16-token pages, fp32 logits over 128256): one rgd_decode_step, i.e. the
shared-prefix split-KV attention, then the sample head (argmax / temperature +
min-p + Philox draw) with the trie gate fused in.  Inputs are seeded synthetic
data resident in HBM; L2 is evicted (a 256 MiB write, then a 320 MiB read)
before every timed step, outside the timed events.  Extra keys time the
long-prompt and high-batch steps, the largest head and gate sweeps, the whole
128-step gated loop, the soft gate and the residual precheck.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Prints one JSON line (rank 0).  ``--impl reference`` times the CPU oracle on the
host cores on a bounded sample of the same workload.  Under torchrun (N > 1)
every rank runs its own batch (weak scaling, no collective in the data path).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

os.environ.setdefault("OMP_NUM_THREADS", "1")
os.environ.setdefault("OPENBLAS_NUM_THREADS", "1")
os.environ.setdefault("MKL_NUM_THREADS", "1")

import numpy as np  # noqa: E402

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "decode-step rows/sec and achieved HBM GB/s (% of GB300 peak), 1 GPU"
UNIT = "rows/s"
WORKLOAD = ("llama8b-shaped decode step: 16 prompts x (1 probe + 4 sample rows), prompt len U[512,2048], "
            "suffix len U[0,256], 32 q / 8 kv heads, head dim 128, bf16 KV in 16-token pages, "
            "fp32 Zipf(1.1) logits over 128256, T in {1,1.5,2,3}, min-p in {0.05,0.1}, 64 refusal seqs")
FALLBACK_HBM_GBS = 6800.0


def _peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def algorithmic_bytes(case):
    """Bytes the method must read per step: prompt KV once per active group (all kv
    heads), suffix KV once per active row, logits once per active row."""
    a, h = case.attn, case.head
    kv_tok = a.num_kv_heads * 2 * a.head_dim * 2
    rpg = a.rows_per_group
    attn = 0
    for g in range(a.num_groups):
        if a.row_active[g * rpg:(g + 1) * rpg].any():
            attn += int(a.prompt_len[g]) * kv_tok
    attn += int(sum(int(a.suffix_len[r]) * kv_tok for r in range(a.num_rows) if a.row_active[r]))
    es = 4 if h.dtype == "f32" else 2
    head = int(h.row_active.sum()) * h.vocab * es
    return attn, head


# DRAM traffic of one attention launch on the Llama-3-8B-shaped step
# (dram__bytes_read.sum + dram__bytes_write.sum), from one ncu capture of the
# kernel sources whose hash is given (profiles/attn_t_kernel_llama8b.md has the
# command); reported only while those sources are unchanged, else null.
ATTN_TRAFFIC = {"sources_sha256": "adc56870d915", "bytes_per_launch": 121346048}
ATTN_SOURCES = ("attention.cu", "attention_t.cuh")


def _kernel_hash():
    h = hashlib.sha256()
    for f in ATTN_SOURCES:
        h.update(open(os.path.join(ROOT, "paper_2607_20791_gb300", "csrc", f), "rb").read())
    return h.hexdigest()[:12]


def _profiled_traffic():
    """Per-launch DRAM bytes of the attention kernel recorded above, if they
    were taken on the current kernel sources (else None)."""
    if ATTN_TRAFFIC["bytes_per_launch"] is None or ATTN_TRAFFIC["sources_sha256"] != _kernel_hash():
        return None
    return int(ATTN_TRAFFIC["bytes_per_launch"])


class ClockSampler:
    """nvidia-smi clock / throttle-reason samples while the timed region runs.

    The sampler starts a little before the region and stops a little after it;
    `region()` marks the region itself, and the summary keeps only the samples
    whose timestamps fall inside it (all samples, said so, if none does)."""

    FIELDS = ("index,timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    INTERVAL_MS = 100

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None
        self.t0 = self.t1 = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", str(self.INTERVAL_MS)], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        time.sleep(0.2)
        return self

    def start(self):
        self.t0 = time.time()

    def stop(self):
        self.t1 = time.time()

    def __exit__(self, *exc):
        time.sleep(0.2)
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        rows = []
        try:
            for line in open(self.path):
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 10:
                    rows.append(parts)
        except OSError:
            pass
        finally:
            try:
                os.unlink(self.path)
            except OSError:
                pass
        return summarise_clock_rows(rows, self.t0, self.t1)


def _sample_time(stamp: str):
    """nvidia-smi's timestamp (local time, 'YYYY/MM/DD HH:MM:SS.mmm') as epoch seconds, or None."""
    import datetime
    for fmt in ("%Y/%m/%d %H:%M:%S.%f", "%Y/%m/%d %H:%M:%S"):
        try:
            return datetime.datetime.strptime(stamp.strip(), fmt).timestamp()
        except ValueError:
            continue
    return None


def summarise_clock_rows(rows, t0=None, t1=None, slack_s: float = 0.03):
    """Median SM clock, the maximum, and the throttle reasons seen, over the
    samples taken inside [t0, t1] (epoch seconds, with a little slack for the
    sampling interval); over all samples when none falls inside."""
    if not rows:
        return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no nvidia-smi samples"], "samples": 0}
    inside = rows
    scope = "all samples"
    if t0 is not None and t1 is not None:
        sel = [r for r in rows if (lambda t: t is not None and t0 - slack_s <= t <= t1 + slack_s)(_sample_time(r[1]))]
        if sel:
            inside, scope = sel, "timed region"
        else:
            scope = "all samples (none inside the timed region)"

    def num(x):
        try:
            return float(x)
        except ValueError:
            return None

    sm = [num(r[2]) for r in inside if num(r[2]) is not None]
    smax = [num(r[3]) for r in rows if num(r[3]) is not None]
    reasons = set()
    for r in inside:
        for name, col in (("hw_slowdown", 6), ("hw_thermal_slowdown", 7), ("sw_thermal_slowdown", 8),
                          ("sw_power_cap", 9)):
            if r[col].lower().startswith("active"):
                reasons.add(name)
    return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
            "reasons": sorted(reasons), "samples": len(inside), "scope": scope}


def clocks_rejected(clocks) -> bool:
    """A timed region whose clock record shows a hardware or thermal slowdown,
    or SM clocks well below their maximum with no reason (a leftover clock
    lock), is not a valid measurement; a power cap alone is kept."""
    reasons = set(clocks.get("reasons") or [])
    if reasons & {"hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown"}:
        return True
    sm, smax = clocks.get("sm_mhz"), clocks.get("sm_max_mhz")
    return bool(sm and smax and sm < 0.85 * smax and "sw_power_cap" not in reasons)


def measure_with_clock_check(run_region, sync, clock, barrier=None, allreduce_max=None):
    """Runs `run_region()` (the timed region) inside a clock sampler, bracketed
    by `barrier` (all ranks) and `sync` (the device); when the clock record is
    rejected on any rank (`allreduce_max` takes the max of a float over the
    ranks), every rank runs the region once more.  Returns (the region's
    result, the clock summary, whether it was measured again)."""
    remeasured = False
    for attempt in range(2):
        if barrier is not None:
            barrier()
        sync()
        with clock() as clk:
            clk.start()
            result = run_region()
            sync()
            clk.stop()
        if barrier is not None:
            barrier()
        clocks = clk.summary()
        redo = 1.0 if clocks_rejected(clocks) else 0.0
        if allreduce_max is not None:
            redo = allreduce_max(redo)  # every rank measures again, or none
        if attempt == 0 and redo > 0:
            remeasured = True
            continue
        break
    return result, clocks, remeasured


def _dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def aggregate_over_ranks(step_ms: float, e2e_ms: float, attn_ms: float, rows_per_step: int, world: int,
                         device="cpu"):
    """Max of the per-rank times over the job (every rank gets the same
    result), and the whole-job throughputs: world * rows / max step time.
    Needs an initialised process group when world > 1 (NCCL on the GPUs, gloo
    in the CPU tests)."""
    import torch
    vals = torch.tensor([step_ms, e2e_ms, attn_ms], dtype=torch.float64, device=device)
    if world > 1:
        import torch.distributed as dist
        dist.all_reduce(vals, op=dist.ReduceOp.MAX)
    step_ms, e2e_ms, attn_ms = [float(x) for x in vals.tolist()]
    return {"step_ms": step_ms, "e2e_ms": e2e_ms, "attn_ms": attn_ms,
            "value": world * rows_per_step / (step_ms / 1e3), "e2e_value": world * rows_per_step / (e2e_ms / 1e3)}


# ---------------------------------------------------------------------------
# CPU oracle timing (cpu_baseline leg and --impl reference)
# ---------------------------------------------------------------------------
def _oracle_step(case, groups):
    from oracle import attention as oattn
    from oracle import gate as ogate
    from oracle import sampling as osamp
    rpg = case.attn.rows_per_group
    rows = [g * rpg + i for g in groups for i in range(rpg)]
    oattn.decode_attention_case(case.attn, rows=rows)
    res = osamp.sample_head(case.head.logits, case.head.dtype, case.head.is_probe, case.head.temperature,
                            case.head.min_p, case.head.seed, case.head.step, case.head.row_active, rows=rows)
    probe = np.array([[res.tokens[g * rpg]] for g in groups], np.int32)
    ogate.run_gate(probe, case.gate.refusal_seqs, case.gate.eos, case.gate.max_len)
    return len(rows)


def cpu_baseline(case, budget_s: float = 10.0):
    """The oracle as it stands, single-threaded, on whole prompt groups of the step
    until about `budget_s` seconds of CPU work; rows/s scaled from that sample."""
    t0 = time.perf_counter()
    rows = 0
    n = 0
    G = case.attn.num_groups
    while time.perf_counter() - t0 < budget_s:
        rows += _oracle_step(case, [n % G])
        n += 1
    dt = time.perf_counter() - t0
    return {"value": rows / dt, "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": f"{n} prompt groups of the step ({n / G:.1f} passes over its {G} groups, {rows} rows), "
                      f"fp64 NumPy, {dt:.1f} s"}


def run_reference(args):
    world, rank, _ = _dist_env()
    if rank != 0:
        return
    from paper_2607_20791_gb300 import workloads
    case = workloads.llama8b(seed=0)
    G = case.attn.num_groups
    for i in range(args.warmup):
        _oracle_step(case, [i % G])
    times, rows = [], 0
    for i in range(args.steps):
        t0 = time.perf_counter()
        rows += _oracle_step(case, [i % G])
        times.append(time.perf_counter() - t0)
    total = sum(times)
    value = rows / total
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * total / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic",
            "config": {"workload": WORKLOAD, "sample": "one prompt group (5 rows) of the step per timed step"},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle",
                             "sample": "one prompt group (5 rows) per step, fp64 NumPy oracle, single thread"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------
class Evictor:
    """Empties L2 of the next timed call's inputs, outside the timed events: a
    256 MiB write, then a read of 320 MiB (more than twice the 129 MB L2), so
    that the lines left in L2 are clean and the timed call pays no write-back
    of the eviction traffic.  ``clean=False`` stops after the write (then up
    to an L2 of dirty lines is written back inside the timed region)."""

    def __init__(self, dev):
        import torch
        self.w = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
        self.r = torch.ones((320 << 20) // 8, dtype=torch.int64, device=dev)
        self.sink = torch.empty((), dtype=torch.int64, device=dev)

    def __call__(self, clean: bool = True):
        import torch
        self.w.fill_(1)
        if clean:
            torch.sum(self.r, dim=0, out=self.sink)


class StepOnDevice:
    """One decode step's buffers on the device and its calls: rgd_decode_step
    (attention, then the sample head with the gate fused in), its two halves
    apart, and the reset of the state the gate changes (gate states and row
    mask back to the step's start), run outside the timed events."""

    def __init__(self, case, dev, kv=None):
        import torch
        from paper_2607_20791_gb300 import binding, device
        self.case = case
        self.att = device.attn_to_device(case.attn, device=dev, kv=kv)
        self.head = device.head_to_device(case.head, device=dev)
        self.trie = binding.Trie(case.gate.refusal_seqs, case.gate.min_confirm)
        self.G, self.rpg = case.attn.num_groups, case.attn.rows_per_group
        self.gstate = binding.new_gate_state(self.G, device=dev)
        self.ra0 = self.att.row_active.clone()
        self.status = torch.zeros(1, dtype=torch.int32, device=dev)

    def reset(self, s):
        from paper_2607_20791_gb300 import binding
        binding.rgd_gate_state_init(self.gstate, self.G, stream=s)
        self.att.row_active.copy_(self.ra0)

    def step(self, s):
        from paper_2607_20791_gb300 import binding
        a, h, g = self.att, self.head, self.case.gate
        binding.rgd_decode_step(a.shape, a.q, a.k_pages, a.v_pages, a.prompt_block_table, a.prompt_len,
                                a.suffix_block_table, a.suffix_len, a.softmax_scale, a.out, a.lse, a.workspace,
                                h.logits, h.is_probe, h.temperature, h.min_p, h.seed, h.step, a.row_active,
                                h.token_out, h.kept_count, self.trie, g.eos, g.max_len, self.gstate, self.status,
                                stream=s)

    def attn(self, s):
        from paper_2607_20791_gb300 import binding
        a = self.att
        binding.rgd_prefix_decode_attn(a.shape, a.q, a.k_pages, a.v_pages, a.prompt_block_table, a.prompt_len,
                                       a.suffix_block_table, a.suffix_len, a.row_active, a.softmax_scale, a.out,
                                       a.lse, a.workspace, self.status, stream=s)

    def head_gate(self, s, g0=0, g1=None):
        """The gated head over groups [g0, g1) (all by default)."""
        from paper_2607_20791_gb300 import binding
        a, h, g = self.att, self.head, self.case.gate
        g1 = self.G if g1 is None else g1
        r0, r1 = g0 * self.rpg, g1 * self.rpg
        binding.rgd_sample_head_gated(h.logits[r0:r1], h.is_probe[r0:r1], h.temperature[r0:r1], h.min_p[r0:r1],
                                      h.seed[r0:r1], h.step, a.row_active[r0:r1], h.token_out[r0:r1],
                                      h.kept_count[r0:r1], self.trie, self.rpg, g.eos, g.max_len,
                                      self.gstate[g0:g1], self.status, stream=s)

    def close(self):
        self.trie.close()


def _median(xs):
    xs = sorted(xs)
    return xs[len(xs) // 2]


def time_step(sd, stream, evict, n, warmup=3):
    """Graph of one step (timed with events around each replay, L2 evicted and
    state reset before each), then the same number of eager steps with events
    around attention and around the gated head.  Means in ms."""
    import torch
    s = stream.cuda_stream
    with torch.cuda.stream(stream):
        for _ in range(3):
            sd.reset(s)
            sd.step(s)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            sd.step(s)
        torch.cuda.synchronize()
        step_ms, attn_ms, head_ms = [], [], []
        for i in range(warmup + n):
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
            evict()
            sd.reset(s)
            ev[0].record(stream)
            g.replay()
            ev[1].record(stream)
            ev[1].synchronize()
            if i >= warmup:
                step_ms.append(ev[0].elapsed_time(ev[1]))
        for i in range(warmup + n):
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
            evict()
            sd.reset(s)
            ev[0].record(stream)
            sd.attn(s)
            ev[1].record(stream)
            sd.head_gate(s)
            ev[2].record(stream)
            ev[2].synchronize()
            if i >= warmup:
                attn_ms.append(ev[0].elapsed_time(ev[1]))
                head_ms.append(ev[1].elapsed_time(ev[2]))
    mean = lambda x: sum(x) / len(x)
    return g, mean(step_ms), mean(attn_ms), mean(head_ms)


def _device_kv(attn_case, dev, seed):
    """K and V pools ~ N(0, 1) in bf16, drawn on the device (the kernels' time
    does not depend on the values; the parity tests use the seeded host draw)."""
    import torch
    gen = torch.Generator(device=dev)
    gen.manual_seed(seed)
    shape = (attn_case.num_pages, attn_case.num_kv_heads, attn_case.page_size, attn_case.head_dim)
    k = torch.randn(shape, generator=gen, device=dev, dtype=torch.bfloat16)
    v = torch.randn(shape, generator=gen, device=dev, dtype=torch.bfloat16)
    return k, v


def config_leg(name, case, dev, stream, evict, n, peak):
    """Throughput and HBM roofline fraction of one more configuration's step."""
    import torch
    sd = StepOnDevice(case, dev, kv=_device_kv(case.attn, dev, seed=7))
    _, step_ms, attn_ms, head_ms = time_step(sd, stream, evict, n)
    attn_b, head_b = algorithmic_bytes(case)
    status = int(sd.status.item())
    rows = int(case.head.row_active.sum())
    sd.close()
    del sd
    torch.cuda.empty_cache()
    gbs = lambda b, ms: b / (ms / 1e3) / 1e9
    return {"workload": name, "rows_per_step": rows, "ms_per_step": step_ms, "rows_per_s": rows / (step_ms / 1e3),
            "attention_ms": attn_ms, "head_gate_ms": head_ms, "attention_bytes": attn_b, "logits_bytes": head_b,
            "step_hbm_frac": gbs(attn_b + head_b, step_ms) / peak,
            "attention_hbm_frac": gbs(attn_b, attn_ms) / peak,
            "head_hbm_frac": gbs(head_b, head_ms) / peak, "dev_status": status}


def sweep_leg(dev, stream, evict, n, peak):
    """The largest head sweep (1024 x 262144, fp32 and bf16; temperatures
    0-10, min-p 0-0.3) and the gate sweep (1024 groups, 1000 refusal
    sequences, 32-token probes), each kernel timed alone."""
    import torch
    from paper_2607_20791_gb300 import binding, device, workloads
    out = {}
    base = workloads.head_sweep(1024, 262144, "f32", seed=11)
    for dt in ("f32", "bf16"):
        hc = base if dt == "f32" else workloads.make_head_case(
            base.name, base.logits, "bf16", base.is_probe, base.temperature, base.min_p, seed=11)
        h = device.head_to_device(hc, device=dev)
        ts = []
        with torch.cuda.stream(stream):
            for i in range(3 + n):
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                evict()
                e0.record(stream)
                h.run(stream=stream.cuda_stream, with_mask=False)
                e1.record(stream)
                e1.synchronize()
                if i >= 3:
                    ts.append(e0.elapsed_time(e1))
        b = hc.rows * hc.vocab * (4 if dt == "f32" else 2)
        ms = sum(ts) / len(ts)
        out[f"head_1024x262144_{dt}"] = {"us": 1e3 * ms, "bytes": b, "hbm_frac": b / (ms / 1e3) / 1e9 / peak,
                                          "dev_status": int(h.dev_status.item())}
        del h
    gc = workloads.gate_sweep(groups=1024, n_seq=1000, vocab=128256, n_steps=32, seed=3)
    trie = binding.Trie(gc.refusal_seqs, 2)
    st = binding.new_gate_state(1024, device=dev)
    toks = torch.from_numpy(gc.tokens).to(dev)
    ts = []
    with torch.cuda.stream(stream):
        for i in range(3 + n):
            binding.rgd_gate_state_init(st, 1024, stream=stream.cuda_stream)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            binding.rgd_probe_gate(trie, 1024, 1, toks, 32, 32, gc.eos, gc.max_len, st, stream=stream.cuda_stream)
            e1.record(stream)
            e1.synchronize()
            if i >= 3:
                ts.append(e0.elapsed_time(e1))
    trie.close()
    out["gate_1024x32_tokens"] = {"us": 1e3 * sum(ts) / len(ts), "note": "32 probe tokens per group in one call"}
    torch.cuda.empty_cache()
    return out


def loop_leg(dev, stream, evict, n):
    """The Llama-3-8B-shaped gated loop (128 steps from the prompt end, one CUDA
    graph; per step the probe tokens are planted in the logits, one
    rgd_decode_step runs, the logits go back and the active rows' suffixes
    grow): time per loop and active rows per second."""
    import torch
    from paper_2607_20791_gb300 import device, workloads
    case = workloads.llama8b_loop(seed=0, with_kv=False)
    case.attn.k_pages, case.attn.v_pages = None, None
    kv = _device_kv(case.attn, dev, seed=8)
    loop = device.DeviceLoop(case, stream, keep_history=False, kv=kv)
    loop.capture()
    ts = []
    with torch.cuda.stream(stream):
        for i in range(2 + n):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            evict()
            e0.record(stream)
            loop.graph.replay()
            e1.record(stream)
            e1.synchronize()
            if i >= 2:
                ts.append(e0.elapsed_time(e1))
    rows = int((loop.tok >= 0).sum().item())  # rows that drew a token, over the loop's steps
    status = int(loop.status.item())
    loop.close()
    ms = sum(ts) / len(ts)
    return {"steps": case.n_steps, "ms_per_loop": ms, "us_per_step": 1e3 * ms / case.n_steps,
            "active_rows_per_loop": rows, "rows_per_s": rows / (ms / 1e3), "dev_status": status,
            "launches_per_step": {"library": 2, "torch (input staging, suffix growth)": 3}}


def run_ours(args):
    import torch
    world, rank, local = _dist_env()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    else:
        torch.cuda.set_device(0)
    dev = torch.device("cuda", torch.cuda.current_device())

    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_20791_gb300 import binding, workloads

    peak, peak_kind = _peaks()
    case = workloads.llama8b(seed=rank)
    attn_bytes, head_bytes = algorithmic_bytes(case)
    step_bytes = attn_bytes + head_bytes
    G, rpg = case.attn.num_groups, case.attn.rows_per_group
    R = G * rpg
    rows_per_step = int(case.head.row_active.sum())
    stream = torch.cuda.Stream(device=dev)
    s = stream.cuda_stream
    evict = Evictor(dev)
    sd = StepOnDevice(case, dev)

    # The step is one CUDA graph of rgd_decode_step (two kernels: attention,
    # then the gated head, scheduled while the attention finishes); the headline
    # is timed on it.  The split into attention and gated head comes from a
    # second pass of as many steps launched eagerly with events around each.
    with torch.cuda.stream(stream):
        for _ in range(3):  # eager warm-up (also sets kernel attributes before capture)
            sd.reset(s)
            sd.step(s)
        torch.cuda.synchronize()
        g_step = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g_step, stream=stream):
            sd.step(s)
        torch.cuda.synchronize()
    launches_per_step = 2  # attention (split jobs merged inside), sample head with the gate fused in

    def one_step():
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
        evict()
        sd.reset(s)
        ev[0].record(stream)
        g_step.replay()
        ev[1].record(stream)
        ev[1].synchronize()
        return ev[0].elapsed_time(ev[1])

    def split_step():
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
        evict()
        sd.reset(s)
        ev[0].record(stream)
        sd.attn(s)
        ev[1].record(stream)
        sd.head_gate(s)
        ev[2].record(stream)
        ev[2].synchronize()
        return ev[0].elapsed_time(ev[1]), ev[1].elapsed_time(ev[2])

    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            one_step()
            split_step()
        torch.cuda.synchronize()

    def timed_region():
        with torch.cuda.stream(stream):
            s_ms = [one_step() for _ in range(args.steps)]
            sp = [split_step() for _ in range(args.steps)]
        return s_ms, sp

    def max_over_ranks(x: float) -> float:
        t = torch.tensor([x], dtype=torch.float64, device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        return float(t.item())

    (step_ms, split), clocks, remeasured = measure_with_clock_check(
        timed_region, torch.cuda.synchronize, lambda: ClockSampler(torch.cuda.current_device()),
        barrier=dist.barrier if world > 1 else None, allreduce_max=max_over_ranks if world > 1 else None)
    attn_ms = [t[0] for t in split]
    hg_ms = [t[1] for t in split]
    mean_step = sum(step_ms) / len(step_ms)
    mean_attn = sum(attn_ms) / len(attn_ms)
    mean_hg = sum(hg_ms) / len(hg_ms)
    status = int(sd.status.item())
    n_side = max(5, min(args.steps, 100))  # steps of the legs outside the headline

    # ---- the attention after a write-only eviction: the dirty lines it leaves
    # in L2 are written back inside the timed region (context for the headline's
    # clean eviction)
    dirty_ms, clean_ms = [], []
    with torch.cuda.stream(stream):
        for i in range(3 + n_side):
            for clean, acc in ((False, dirty_ms), (True, clean_ms)):
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                evict(clean=clean)
                sd.reset(s)
                e0.record(stream)
                sd.attn(s)
                e1.record(stream)
                e1.synchronize()
                if i >= 3:
                    acc.append(e0.elapsed_time(e1))

    # ---- the residual-stream precheck (App. A): once per prompt, not per step;
    # timed alone on the step's 16 groups (d = 4096 bf16)
    pre = workloads.llama8b_precheck(seed=rank)
    pre_h = torch.from_numpy(pre.h.view(np.int16)).to(dev).view(torch.bfloat16)
    pre_w = torch.from_numpy(pre.w).to(dev)
    pre_st = binding.new_gate_state(G, device=dev)
    pre_prob = torch.empty(G, dtype=torch.float32, device=dev)
    pre_ms = []
    with torch.cuda.stream(stream):
        for i in range(3 + n_side):
            binding.rgd_gate_state_init(pre_st, G, stream=s)
            evict()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            binding.rgd_residual_precheck(pre_h, pre_w, pre.b, pre.theta, rpg, pre_st, None, pre_prob, stream=s)
            e1.record(stream)
            e1.synchronize()
            if i >= 3:
                pre_ms.append(e0.elapsed_time(e1))
    pre_bytes = pre.groups * pre.d * 2 + pre.d * 4 + pre.groups * (4 + 20)

    # ---- the soft compatibility gate (the appendix ablation's Alg. 2): an
    # alternative to the hard gate; timed alone on the step's probe rows from a
    # fresh state (top-K 40, rho 0.1; the step's greedy tokens mostly leave the
    # refusal set, so the soft branch runs)
    head = sd.head
    soft_tok = torch.empty(G, dtype=torch.int32, device=dev)
    soft_ms = []
    with torch.cuda.stream(stream):
        for i in range(3 + n_side):
            binding.rgd_gate_state_init(pre_st, G, stream=s)
            evict()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            binding.rgd_soft_gate(sd.trie, G, rpg, head.logits, rpg * head.logits.shape[1], 40, 0.1, 8,
                                  case.gate.eos, case.gate.max_len, pre_st, soft_tok, stream=s)
            e1.record(stream)
            e1.synchronize()
            if i >= 3:
                soft_ms.append(e0.elapsed_time(e1))
    soft_bytes = G * head.logits.shape[1] * head.logits.element_size()

    # ---- end to end through the public API with host buffers ----------------
    # One CUDA graph per step.  The copy engine takes host-to-device copies one
    # at a time (about 200 GB/s over the host link), so the small inputs
    # (queries, block tables, lengths, sampling parameters) travel as one
    # packed copy -- on the device they are views of one buffer -- and then the
    # 41 MB of logits on a second stream while the attention runs; the gated
    # head runs once the logits are in; the tokens and gate states are read
    # back.  Every input comes from pinned host memory each step.  (Copying
    # the logits in chunks of groups and sampling each chunk as it lands was
    # no faster: the head's time is latency, not rows.)
    att = sd.att
    small_src = [(case.attn.q, att, "q"), (case.attn.prompt_block_table, att, "prompt_block_table"),
                 (case.attn.prompt_len, att, "prompt_len"), (case.attn.suffix_block_table, att, "suffix_block_table"),
                 (case.attn.suffix_len, att, "suffix_len"), (case.attn.row_active, att, "row_active"),
                 (case.head.temperature, head, "temperature"), (case.head.min_p, head, "min_p"),
                 (case.head.seed.view(np.int64), head, "seed"), (case.head.is_probe, head, "is_probe")]
    offs, pack_bytes = [], 0
    for _, obj, name in small_src:
        d = getattr(obj, name)
        offs.append(pack_bytes)
        pack_bytes += (d.numel() * d.element_size() + 255) // 256 * 256
    pack_dev = torch.empty(pack_bytes, dtype=torch.uint8, device=dev)
    pack_host = torch.zeros(pack_bytes, dtype=torch.uint8).pin_memory()
    replaced = []  # the step's earlier input tensors, kept alive (the step's graph points at them)
    for (a, obj, name), off in zip(small_src, offs):
        d = getattr(obj, name)
        nb = d.numel() * d.element_size()
        hb = np.ascontiguousarray(a).view(np.uint8).reshape(-1)
        assert hb.size == nb, name
        pack_host[off:off + nb].copy_(torch.from_numpy(hb))
        view = pack_dev[off:off + nb].view(d.dtype).view(d.shape)
        view.copy_(d)
        replaced.append(d)
        setattr(obj, name, view)
    logits_dev = head.logits
    logits_pin = torch.from_numpy(np.ascontiguousarray(case.head.logits))
    if logits_pin.dtype != logits_dev.dtype:
        logits_pin = logits_pin.view(logits_dev.dtype)
    logits_pin = logits_pin.reshape(logits_dev.shape).pin_memory()
    h2d_bytes = pack_bytes + logits_pin.numel() * logits_pin.element_size()
    tok_host = torch.empty(R, dtype=torch.int32).pin_memory()
    st_host = torch.empty_like(sd.gstate, device="cpu").pin_memory()
    d2h_bytes = tok_host.numel() * 4 + st_host.numel()
    side = torch.cuda.Stream(device=dev)

    def e2e_body():
        pack_dev.copy_(pack_host, non_blocking=True)
        side.wait_stream(stream)  # (the logits queue behind the packed copy, not ahead of it)
        with torch.cuda.stream(side):
            logits_dev.copy_(logits_pin, non_blocking=True)
        sd.attn(s)
        stream.wait_stream(side)
        sd.head_gate(s)
        tok_host.copy_(head.token_out, non_blocking=True)
        st_host.copy_(sd.gstate, non_blocking=True)

    with torch.cuda.stream(stream):
        sd.reset(s)
        e2e_body()
        torch.cuda.synchronize()
        g_e2e = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g_e2e, stream=stream):
            e2e_body()
        torch.cuda.synchronize()
        e2e_list = []
        for i in range(args.warmup + args.steps):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            evict()
            binding.rgd_gate_state_init(sd.gstate, G, stream=s)
            e0.record(stream)
            g_e2e.replay()
            e1.record(stream)
            e1.synchronize()
            if i >= args.warmup:
                e2e_list.append(e0.elapsed_time(e1))
    e2e_ms = sum(e2e_list) / len(e2e_list)

    # ---- size-matched copy (context for the roofline fraction) ------------------
    # a plain device copy moving the attention's algorithmic byte count (half read,
    # half written), timed like the kernels after each eviction: the bandwidth a
    # transfer of this size reaches at all
    half = (attn_bytes // 2 + 15) // 16 * 16
    c_src = torch.ones(half, dtype=torch.uint8, device=dev)
    c_dst = torch.empty_like(c_src)
    copy_res = {}
    with torch.cuda.stream(stream):
        for clean in (True, False):
            ts = []
            for i in range(12):
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                evict(clean=clean)
                a.record(stream)
                c_dst.copy_(c_src)
                b.record(stream)
                b.synchronize()
                if i >= 3:
                    ts.append(a.elapsed_time(b))
            copy_res[clean] = _median(ts)
    del c_src, c_dst
    copy_ms = copy_res[True]

    # ---- the other configurations (rank 0 only: extra keys, not the headline)
    legs = {}
    if rank == 0:
        legs["long_prompt"] = config_leg(
            "4 prompts x 32768 tokens, 1 probe + 8 sample rows, suffix U[0,1024], 64 q / 8 kv heads, D 128, "
            "bf16 logits over 128256, T 2, min-p 0.05", workloads.long_prompt(seed=0, with_kv=False), dev, stream,
            evict, n_side, peak)
        legs["high_batch"] = config_leg(
            "256 prompts, lengths log-normal (median 1024, sigma 1, 128-8192), 1 probe + 1 sample row, 30 % of "
            "groups' sample rows off, 32 q / 8 kv heads, D 128, bf16 logits over 152064",
            workloads.high_batch(seed=0, with_kv=False), dev, stream, evict, n_side, peak)
        legs["sweep"] = sweep_leg(dev, stream, evict, n_side, peak)
        legs["gated_loop"] = loop_leg(dev, stream, evict, max(3, min(args.steps, 10)))

    # ---- max over ranks --------------------------------------------------------
    agg = aggregate_over_ranks(mean_step, e2e_ms, mean_attn, rows_per_step, world, device=dev)
    mean_step, e2e_ms, mean_attn = agg["step_ms"], agg["e2e_ms"], agg["attn_ms"]
    value, e2e_value = agg["value"], agg["e2e_value"]

    if rank == 0:
        attn_gbs = attn_bytes / (mean_attn / 1e3) / 1e9
        step_gbs = step_bytes / (mean_step / 1e3) / 1e9
        traffic = _profiled_traffic()
        cpu = cpu_baseline(case) if world == 1 else None
        clocks["remeasured"] = remeasured
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": mean_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": WORKLOAD, "rows_per_step": rows_per_step, "groups": G,
                       "l2": "evicted before every timed step, outside the timed events: a 256 MiB write, then a "
                             "320 MiB read, so that L2 holds only clean lines of other data",
                       "timing": "CUDA events per step on the launching stream around one CUDA graph of "
                                 "rgd_decode_step (attention, then the sample head with the gate fused in); gate "
                                 "states and row mask reset before each step outside the events; kernels_ms and "
                                 "roofline from a second pass of as many steps launched eagerly with events around "
                                 "each kernel",
                       "parallelism": f"replicas x{world}"},
            "step_hbm_gbs": step_gbs, "step_hbm_frac": step_gbs / peak,
            "step_algorithmic_bytes": step_bytes,
            "kernels_ms": {"attention": mean_attn, "sample_head_with_gate": mean_hg},
            "roofline": {"bound": "hbm", "kernel": "attn_t_kernel<128, 3>", "achieved": attn_gbs,
                         "peak": peak, "unit": "GB/s", "frac": attn_gbs / peak, "traffic": traffic,
                         "traffic_source": ("one ncu capture of these kernel sources (dram bytes read + written per "
                                            "launch), recorded in bench.py with the sources' hash"
                                            if traffic is not None else
                                            "none: no ncu capture of the current kernel sources"),
                         "algorithmic_bytes": attn_bytes, "peak_source": peak_kind},
            "cpu_baseline": cpu,
            "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d_bytes,
                    "d2h_bytes_per_step": d2h_bytes, "ms_per_step": e2e_ms,
                    "note": "one CUDA graph per step: the small inputs as one packed copy, then the logits on a "
                            "second stream while the attention runs; the gated head after both"},
            "gpu_launches": launches_per_step * args.steps,
            "split_pass_launches": launches_per_step * args.steps,
            "attention_after_write_only_eviction_ms": sum(dirty_ms) / len(dirty_ms),
            "attention_after_clean_eviction_ms": sum(clean_ms) / len(clean_ms),
            "soft_gate": {"us": 1e3 * _median(soft_ms), "groups": G, "bytes": soft_bytes,
                          "gbs": soft_bytes / (_median(soft_ms) / 1e3) / 1e9,
                          "note": "alternative to the hard gate (top-K 40, rho 0.1), outside the step"},
            "residual_precheck": {"us": 1e3 * _median(pre_ms), "groups": pre.groups, "d": pre.d,
                                  "bytes": pre_bytes, "bound": "launch latency (a d + 1 logistic readout)",
                                  "note": "once per prompt, outside the step"},
            "copy_ceiling": {"bytes": 2 * half, "us": copy_ms * 1e3, "gbs": 2 * half / (copy_ms / 1e3) / 1e9,
                             "frac_of_peak": 2 * half / (copy_ms / 1e3) / 1e9 / peak,
                             "attention_frac_of_copy": copy_ms / mean_attn,
                             "after_write_only_eviction_us": copy_res[False] * 1e3,
                             "note": "a plain device copy of the attention's algorithmic byte count (half read, "
                                     "half written), L2 evicted as for the step, median of 9: what a transfer of "
                                     "this size reaches"},
            "configs": legs,
            "clocks": clocks, "dev_status": status,
        }
        print(json.dumps(line), flush=True)
    sd.close()
    if world > 1:
        dist.destroy_process_group()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None,
                    help="timed steps (default 2000 on the GPU, ~0.6 s; 300 for the CPU reference arm, ~11 s)")
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    args = ap.parse_args()
    if args.steps is None:
        args.steps = 2000 if args.impl == "ours" else 300
    args.warmup = max(3, args.warmup)
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
