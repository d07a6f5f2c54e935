"""Decode-step benchmark of libegmla on synthetic EG-MLA workloads.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload c32k] [--impl reference]
    python bench.py --sweep        (decode throughput vs context length)
    python bench.py --workload layers24_full   (24 whole attention layers per step)
    python bench.py --workload prefill         (prompt processing: 8 prompts x 4096 tokens)

A step is one pass of the whole decode hot path for one batch: append of each
sequence's new token to the paged latent cache, query absorption, the split-KV
gated latent attention and the split merge with the W_UV up-projection (for
layers24: that, for each of 24 attention layers in turn).  The default
workload is the 32K-context one (batch 8, 16 heads, d_c 256, RoPE 64, 64-token
pages permuted over a shared pool, vocabulary 32000), on which the roofline
target of the hot path is stated.  --sweep prints one line per context length
L = 1K .. 64K at batch 8 (d_c 256, contiguous pages).

value: decode tokens/s (new tokens produced per second, all GPUs) with every
input resident in HBM; the step is replayed from a CUDA graph over three
rotating cache replicas (3 x 168 MB > L2; layers24: 24 distinct layer caches),
so the latent stream comes from HBM.
e2e: the same metric through the C ABI from pinned HOST buffers, the per-step
inputs (packed in one buffer) copied in and the output copied back inside the
timed region, calls issued eagerly from Python.
roofline: the decode kernel's latent-cache bytes per launch divided by its own
CUDA-event duration (events recorded around every decode launch inside a
captured graph of the same steps, on the launching stream), against the
measured HBM copy bandwidth.
cpu_baseline / --impl reference: the fp64 oracle on the host cores on a bounded
sample of the same workload, scaled to decode tokens/s.

prefill / prefill_ragged: a step is one eg_mla_prefill call over the packed
prompts (gate + LayerNorm and cache write per token, the per-head key/value
up-projection, causal attention); value = prompt tokens/s, the roofline is the
attention kernel's causal FLOPs over its own CUDA-event time against the bf16
tensor peak, e2e copies the prompts' q, c, k^R and ids in from pinned host
memory and the output back every step, and the oracle baseline times whole
heads of the first prompt.

Multi-GPU (torchrun): every rank runs its own replica of the workload (the
sequences are independent; no data-path collective); the slowest rank's time
sets the aggregate.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time


def host_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


# The fp64 oracle's matrix products run in the BLAS numpy loads; its thread
# count is pinned here, before numpy is imported, so that the CPU baseline can
# state the threads it used (an explicit setting by the caller is kept).
BLAS_ENV = ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS")
for _v in BLAS_ENV:
    os.environ.setdefault(_v, str(host_cores()))
BLAS_THREADS = int(os.environ["OPENBLAS_NUM_THREADS"])

import numpy as np  # noqa: E402

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "decode tokens/sec and latent-cache HBM GB/s (fraction of ~8 TB/s) vs ctx len"
UNIT = "tokens/s"
REPLICAS = 3


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None,
                    help="timed steps (default 20000; 200 for layers24, 2000 per length for --sweep)")
    ap.add_argument("--warmup", type=int, default=30)
    ap.add_argument("--workload", default="c32k",
                    choices=["c32k", "c32k_embed", "c4k", "ragged", "ragged_mla", "layers24", "layers24_full", "r0",
                             "prefill", "prefill_ragged"])
    ap.add_argument("--sweep", action="store_true",
                    help="decode throughput vs context length: batch 8, d_c 256, L = 1K .. 64K, one line per L")
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--splits", type=int, default=0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--layers", type=int, default=0,
                    help="layers of the layers24 / layers24_full workloads (default 24; fewer for a profiling run)")
    ap.add_argument("--e2e-steps", type=int, default=0)
    ap.add_argument("--oracle-probe", default=None, help=argparse.SUPPRESS)
    ap.add_argument("--oracle-budget", type=float, default=4.0, help=argparse.SUPPRESS)
    ap.add_argument("--no-mla-baseline", action="store_true",
                    help="skip the gate-off (plain MLA) measurement of the same workload")
    ap.add_argument("--lgz", type=int, default=1,
                    help="layers24_full: layer group size (consecutive layers share one latent cache and its "
                         "KV projection, Appendix H)")
    return ap.parse_args()


def synth_mod():
    from paper_2509_16686_gb300 import synth
    return synth


def make_workload(name):
    from paper_2509_16686_gb300 import synth
    if name == "c32k":
        case = synth.case_c32k(keep_logical=False)
        desc = "c32k: batch 8 x context 32768, 16 heads, d_nope 128, d_rope 64, d_c 256, vocab 32000, " \
               "64-token pages permuted over one pool, uniform ids"
    elif name == "c32k_embed":
        case = synth.case_c32k(keep_logical=False)
        desc = "c32k_embed: the c32k step with its gate table computed in the step from the gate embedding " \
               "(eg_mla_gate_table: E [32000 x 256] W^UE^T, then eg_mla_step), the EG-MLA form without a stored table"
    elif name == "c4k":
        case = synth.case_c4k(keep_logical=False)
        desc = "c4k: batch 32 x context 4096, 16 heads, d_c 256, d_rope 64, vocab 32000, contiguous pages"
    elif name == "ragged":
        case = synth.case_ragged(keep_logical=False)
        desc = "ragged: batch 128, contexts log-uniform [128, 16384], 16 heads, d_c 192, vocab 50000, Zipf(1.1) ids"
    elif name == "ragged_mla":
        case = synth.case_ragged(gate=False, keep_logical=False)
        desc = "ragged_mla: plain-MLA baseline (gate off) at d_c 512 on the ragged lengths"
    elif name == "layers24_full":
        case = synth.case_layer(0)
        desc = f"layers24_full: decoder step over {layers_of(name)} full attention layers (hidden 2048: W^Q and W^DKV,KR " \
               "projections in this library's tcgen05 GEMM, fused kv_norm + RoPE, append, gated latent attention, W^O; " \
               "each layer's output is the next layer's input), batch 64 x context 8192, 16 heads, d_c 256, " \
               "d_rope 64, vocab 50000, contiguous pages; layer 0's seeded synthetic cache, ids, gate table and " \
               f"weights cloned into {layers_of(name)} distinct device copies"
    elif name == "layers24":
        case = synth.case_layer(0)
        desc = f"layers24: decoder step over {layers_of(name)} attention layers (append + decode per layer on one stream), " \
               "batch 64 x context 8192, 16 heads, d_c 256, d_rope 64, vocab 50000, contiguous pages; layer 0's " \
               f"seeded synthetic cache, ids, gate table, weights and inputs cloned into {layers_of(name)} distinct " \
               "device copies"
    else:
        ctx = int(name[3:])
        case = synth.case_c4k(batch=8, ctx=ctx, keep_logical=False)
        desc = f"ctx{ctx}: batch 8 x context {ctx}, 16 heads, d_c 256, d_rope 64, vocab 32000, contiguous pages"
    return case, desc


LAYERS_OVERRIDE = None   # --layers: fewer layers for a profiling run of the layer workloads


def layers_of(name):
    if not name.startswith("layers24"):
        return 1
    return LAYERS_OVERRIDE or 24


SWEEP_CTX = (1024, 2048, 4096, 8192, 16384, 32768, 65536)


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def max_over_ranks(ms, dist, device):
    """The slowest rank's time (every rank gets it); `ms` itself without a process group."""
    if dist is None:
        return ms
    import torch
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def algorithmic_bytes(case, cache_bytes):
    """Bytes one decode launch must move at least: the latent-cache stream
    (c^KV, k^R and the token id of every cached token), each distinct gate row
    G[id] once (the ids of the cached tokens after the step's append), and
    W_UV of every head.  Queries, outputs, split partials and LayerNorm
    parameters (under 1 % here) are left out."""
    d = case.dims
    elem = 2 if d.dtype == "bf16" else 4
    gate_rows = 0
    if d.gate:
        P = d.page_size
        ids = []
        for b in range(case.batch):
            L = int(case.seq_lens[b])
            if L == 0:
                continue
            pages = case.block_table[b, :(L + P - 1) // P]
            ids.append(case.id_pool[pages].reshape(-1)[:L - 1])
            ids.append(case.ids_new[b:b + 1])
        gate_rows = int(np.unique(np.concatenate(ids)).size) * d.d_c * elem if ids else 0
    w_uv = d.num_heads * d.d_v * d.d_c * elem
    return {"cache": int(cache_bytes), "gate_rows_unique": gate_rows, "w_uv": w_uv,
            "total": int(cache_bytes) + gate_rows + w_uv}


def whole_job_rate(world_size, batch, steps, ms):
    """Decode tokens/s of the whole job: every rank decodes `batch` sequences per
    step (weak scaling), `steps` steps in `ms` milliseconds (the slowest rank's)."""
    return world_size * batch * steps / (ms / 1e3)


# ----------------------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id):
        self.gpu_id = gpu_id
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                                          "-lms", "100", "-i", str(self.gpu_id)], stdout=subprocess.PIPE,
                                         stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.25)
        return self

    def __exit__(self, *a):
        self.lines = []
        if self.proc is not None:
            time.sleep(0.15)
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                out, _ = self.proc.communicate()
            self.lines = [l for l in out.splitlines() if l.strip()]

    def summary(self):
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for l in self.lines:
            f = [x.strip() for x in l.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm)}


def nvsmi_id(torch, dev):
    try:
        u = str(torch.cuda.get_device_properties(dev).uuid)
        return u if u.startswith("GPU-") else "GPU-" + u
    except Exception:
        return dev


# ----------------------------------------------------------------------------- CPU oracle timing
def oracle_sample_rate(case, budget_s):
    """Decode tokens/s of the fp64 oracle on host cores, from a bounded sample:
    whole heads of whole sequences while the budget lasts (at least one head)."""
    from oracle import egmla_oracle as orc
    B, H = case.batch, case.dims.num_heads
    t0 = time.perf_counter()
    heads_done = 0
    b = 0
    while True:
        for h in range(H):
            orc.decode_unabsorbed(case, batches=[b], heads=[h])
            heads_done += 1
            if time.perf_counter() - t0 > budget_s:
                break
        if time.perf_counter() - t0 > budget_s or b + 1 >= B:
            break
        b += 1
    dt = time.perf_counter() - t0
    # one decode token = all heads of one sequence
    rate = (heads_done / H) / dt
    sample = f"{heads_done} head(s) of {b + 1} sequence(s) at full context, {dt:.1f} s"
    return rate, sample, dt


def oracle_rate_subprocess(workload, threads, budget_s):
    """The oracle's decode tokens/s on `workload` in a child process whose BLAS
    runs `threads` threads (the single-thread times of the baseline)."""
    env = dict(os.environ)
    for v in BLAS_ENV:
        env[v] = str(threads)
    r = subprocess.run([sys.executable, os.path.abspath(__file__), "--oracle-probe", workload,
                        "--oracle-budget", str(budget_s)], capture_output=True, text=True, env=env, timeout=600)
    if r.returncode != 0:
        return {"error": r.stderr.strip().splitlines()[-1:] if r.stderr else "failed"}
    return json.loads(r.stdout.strip().splitlines()[-1])


def oracle_probe(workload, budget_s):
    """(child process) one bounded oracle sample of a workload, as JSON."""
    from paper_2509_16686_gb300 import synth
    case = synth.case_tiny() if workload == "tiny" else make_workload(workload)[0]
    rate, sample, dt = oracle_sample_rate(case, budget_s)
    print(json.dumps({"value": rate, "sample": sample, "seconds": dt, "threads": BLAS_THREADS}))
    return 0


def cpu_baseline_line(case, budget_s, n_layers=1):
    """cpu_baseline: the oracle on this process's BLAS threads over a bounded
    sample of the workload, plus single-thread rates on the tiny fp32 and the
    4K workloads."""
    rate, sample, _ = oracle_sample_rate(case, budget_s)
    if n_layers > 1:
        rate /= n_layers
        sample += f", one layer of {n_layers} (rate / {n_layers})"
    single = {w: oracle_rate_subprocess(w, 1, 4.0) for w in ("tiny", "c4k")}
    return {"value": rate, "unit": UNIT, "cores": BLAS_THREADS, "threads": BLAS_THREADS, "host_cores": host_cores(),
            "kind": "oracle", "sample": sample,
            "single_thread": {w: {"value": v.get("value"), "unit": UNIT, "sample": v.get("sample")}
                              for w, v in single.items()}}


def run_reference(args):
    """The reference arm: the fp64 oracle on the host cores.  Each step computes one
    head of sequence 0 over its first S cached tokens, S chosen so that the whole
    run fits in about two minutes; the oracle's cost is linear in the context, so
    the step time is scaled by (L / S) x heads to one decode token."""
    import dataclasses
    ws, rank, _ = dist_env()
    if rank != 0:
        return 0
    if args.workload.startswith("prefill"):
        return run_reference_prefill(args)
    case, desc = make_workload(args.workload)
    from oracle import egmla_oracle as orc
    H = case.dims.num_heads
    L = int(case.seq_lens[0])
    n_steps = max(1, args.steps if args.steps is not None else 10) + max(0, args.warmup)
    probe = dataclasses.replace(case, seq_lens=case.seq_lens[:1].copy(), block_table=case.block_table[:1],
                                q=case.q[:1], c_new=case.c_new[:1], kr_new=case.kr_new[:1],
                                ids_new=case.ids_new[:1])
    t0 = time.perf_counter()
    orc.decode_unabsorbed(probe, batches=[0], heads=[0])
    t_full = time.perf_counter() - t0           # includes the one-time append copy
    t0 = time.perf_counter()
    orc.decode_unabsorbed(probe, batches=[0], heads=[0])
    t_full = min(t_full, time.perf_counter() - t0)
    S = int(min(L, max(64, L * (110.0 / n_steps) / max(t_full, 1e-6))))
    sub = dataclasses.replace(probe, seq_lens=np.array([S], dtype=np.int32))
    orc.appended_pools(sub)
    times = []
    t_start = time.perf_counter()
    for i in range(n_steps):
        t1 = time.perf_counter()
        orc.decode_unabsorbed(sub, batches=[0], heads=[i % H])
        dt = time.perf_counter() - t1
        if i >= args.warmup:
            times.append(dt)
        if time.perf_counter() - t_start > 170:
            break
    n_layers = layers_of(args.workload)
    t_step = statistics.mean(times)
    t_token = t_step * H * (L / S) * n_layers
    rate = 1.0 / t_token
    line = {
        "impl": "reference", "metric": METRIC, "value": rate, "unit": UNIT, "n_gpus": args.gpus,
        "steps": len(times), "warmup": args.warmup, "ms_per_step": t_step * 1e3,
        "ms_per_decode_token_scaled": t_token * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": desc, "batch": case.batch, "ctx": L},
        "cpu_baseline": {"value": rate, "unit": UNIT, "cores": BLAS_THREADS, "threads": BLAS_THREADS,
                         "host_cores": host_cores(), "kind": "oracle",
                         "sample": f"per step one head of one sequence over its first {S} of {L} cached "
                                   f"tokens, scaled x{H} heads x{L / S:.1f} context x{n_layers} layer(s)"
                                   + ("; a whole layer's projections add under 0.2 % to the oracle's "
                                      "attention work per token and are not timed"
                                      if args.workload == "layers24_full" else "")},
        "e2e": {"value": rate, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def run_reference_prefill(args):
    """The reference arm of the prefill workloads: each step is the oracle's
    prefill of one head of the first prompt over its first S tokens (S sized so
    the run ends in about two minutes), scaled by the oracle's quadratic cost
    in the prompt length to all heads and prompts."""
    import dataclasses
    from oracle import egmla_oracle as orc
    pc, desc = prefill_case(args.workload)
    H = pc.dims.num_heads
    L = int(pc.seq_lens[0])
    n_steps = max(1, args.steps if args.steps is not None else 10) + max(0, args.warmup)
    t0 = time.perf_counter()
    orc.prefill(pc, batches=[0], heads=[0])
    t_full = time.perf_counter() - t0
    S = int(min(L, max(64, L * ((110.0 / n_steps) / max(t_full, 1e-6)) ** 0.5)))
    sub = dataclasses.replace(pc, seq_lens=np.array([S], np.int32), cu_seqlens=np.array([0, S], np.int32),
                              q=pc.q[:S], c=pc.c[:S], kr=pc.kr[:S], ids=pc.ids[:S])
    times = []
    t_start = time.perf_counter()
    for i in range(n_steps):
        t1 = time.perf_counter()
        orc.prefill(sub, batches=[0], heads=[i % H])
        dt = time.perf_counter() - t1
        if i >= args.warmup:
            times.append(dt)
        if time.perf_counter() - t_start > 170:
            break
    t_step = statistics.mean(times)
    work = sum(int(x) ** 2 for x in pc.seq_lens) / float(S * S)
    t_call = t_step * H * work
    rate = pc.total_tokens / t_call
    line = {
        "impl": "reference", "metric": "prefill tokens/sec (prompt tokens through gate, cache write, up-projection "
                                      "and causal attention)",
        "value": rate, "unit": "tokens/s", "n_gpus": args.gpus, "steps": len(times), "warmup": args.warmup,
        "ms_per_step": t_step * 1e3, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f64", "data": "synthetic", "config": {"workload": desc, "prompts": pc.batch, "tokens": pc.total_tokens},
        "cpu_baseline": {"value": rate, "unit": "tokens/s", "cores": BLAS_THREADS, "threads": BLAS_THREADS,
                         "host_cores": host_cores(), "kind": "oracle",
                         "sample": f"per step one head of prompt 0 over its first {S} of {L} tokens, scaled x{H} "
                                   f"heads x sum L^2 / S^2 = {work:.1f}"},
        "e2e": {"value": rate, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ----------------------------------------------------------------------------- GPU arm
def kernel_source_sha(files):
    h = hashlib.sha256()
    for f in files:
        path = os.path.join(ROOT, f)
        if not os.path.exists(path):
            return None
        h.update(open(path, "rb").read())
    return h.hexdigest()[:16]


def run_gpu_full_layers(args, workload, torch, dist, ws, rank):
    """The 24-layer decoder step through whole attention layers (eg_mla_layer_decode
    per layer, each layer's output the next one's input)."""
    from oracle import egmla_oracle as orc
    from paper_2509_16686_gb300 import _lib, device, synth
    dev = torch.cuda.current_device()
    case, desc = make_workload(workload)
    lc = synth.make_layer_case(case, 2048, seed=5)
    n_layers = layers_of(workload)
    B, d = case.batch, case.dims
    lgz = max(1, args.lgz)
    if n_layers % lgz:
        raise SystemExit(f"--lgz {lgz} does not divide {n_layers} layers")
    base = device.upload_layer(lc, num_splits=args.splits)
    layers = [base]
    for k in range(1, n_layers):
        if k % lgz:
            # a later layer of a layer group: the group's cache and first-half KV projection
            layer = device.clone_layer(layers[k - k % lgz], share=("workspace", "status", "c_pool", "kr_pool",
                                                                   "id_pool", "block_table"))
            layer.layer_dims = _lib.make_layer_dims(lc.n_embd, lc.rope_theta, lc.rms_eps, share_kv=True)
        else:
            layer = device.clone_layer(base)
        layers.append(layer)
    for k in range(1, n_layers):
        layers[k].x = layers[k - 1].y          # the residual stream is left out: attention layers only
        for name in ("ids_new", "positions", "seq_lens"):   # one step's token ids and lengths, shared
            setattr(layers[k].dc, name, getattr(base.dc, name))
    steps_arg = args.steps if args.steps is not None else 200
    stream = torch.cuda.Stream()
    tokens_cached = int(case.seq_lens.astype(np.int64).sum())
    cache_bytes = tokens_cached * ((d.d_c + d.d_rope) * 2 + 4)
    algo = algorithmic_bytes(case, cache_bytes)
    splits = base.dc.num_splits or _lib.eg_mla_default_num_splits()

    def run_step():
        for layer in layers:
            layer.step(stream)

    with torch.cuda.stream(stream):
        for _ in range(max(3, args.warmup)):
            run_step()
    stream.synchronize()
    assert base.dc.read_status() == 0, "device status after warm-up"
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        run_step()
    with torch.cuda.stream(stream):
        graph.replay()
        graph.replay()
    torch.cuda.synchronize()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(nvsmi_id(torch, dev)) as clk:
        if dist:
            dist.barrier()
        torch.cuda.synchronize()
        with torch.cuda.stream(stream):
            ev0.record(stream)
            for _ in range(steps_arg):
                graph.replay()
            ev1.record(stream)
        torch.cuda.synchronize()
        if dist:
            dist.barrier()
    elapsed_ms = max_over_ranks(ev0.elapsed_time(ev1), dist, "cuda")
    assert base.dc.read_status() == 0, "device status after timed region"
    value = whole_job_rate(ws, B, steps_arg, elapsed_ms)

    # the decode kernel alone, as in run_gpu: events around its launches in a captured step
    _lib.eg_mla_profile_begin(2 * n_layers)
    pgraph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(pgraph, stream=stream):
        run_step()
        run_step()
    with torch.cuda.stream(stream):
        pgraph.replay()
        pgraph.replay()
    stream.synchronize()
    del pgraph
    ms_sum, n_l = _lib.eg_mla_profile_end()
    k_ms = ms_sum / max(1, n_l)
    achieved = algo["total"] / (k_ms * 1e-3) / 1e9
    peaks_path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(peaks_path):
        peak, peak_src = float(json.load(open(peaks_path))["hbm_gbs"]), "measured"
    else:
        peak, peak_src = 6800.0, "fallback"
    gemm = projection_gemm_timing(layers, torch, stream, peak)

    # end to end through the C ABI from pinned host buffers: every step copies in
    # the new tokens' hidden states, ids and positions and reads back the last
    # layer's output
    x0 = base.x.clone()
    base.x = x0
    ins = [x0, base.dc.ids_new, base.dc.positions, base.dc.seq_lens]
    h_ins = [t.cpu().pin_memory() for t in ins]
    h_out = torch.empty(layers[-1].y.shape, dtype=layers[-1].y.dtype).pin_memory()
    e2e_steps = args.e2e_steps or min(steps_arg, 100)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        e0.record(stream)
        for _ in range(e2e_steps):
            for dst, src in zip(ins, h_ins):
                dst.copy_(src, non_blocking=True)
            run_step()
            h_out.copy_(layers[-1].y, non_blocking=True)
        e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1), dist, "cuda")
    assert base.dc.read_status() == 0, "device status after end-to-end run"
    h2d = sum(t.numel() * t.element_size() for t in h_ins)
    d2h = h_out.numel() * h_out.element_size()

    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        t0 = time.perf_counter()
        done = 0
        while done < B and (done == 0 or time.perf_counter() - t0 < 12.0):
            orc.layer_decode(lc, batches=[done])
            done += 1
        dt = time.perf_counter() - t0
        cpu = {"value": done / dt / n_layers, "unit": UNIT, "cores": BLAS_THREADS, "threads": BLAS_THREADS,
               "host_cores": host_cores(), "kind": "oracle",
               "sample": f"the layer oracle on {done} sequence(s) of one layer at full context, {dt:.1f} s "
                         f"(rate / {n_layers} layers)"}
    return {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": steps_arg, "warmup": args.warmup,
        "ms_per_step": elapsed_ms / steps_arg, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16", "data": "synthetic",
        "config": {"workload": desc + (f"; layer groups of {lgz} sharing one cache" if lgz > 1 else ""),
                   "batch": B, "layers": n_layers, "n_embd": 2048, "lgz": lgz,
                   "ctx_tokens_cached": tokens_cached, "splits": splits, "page_size": d.page_size,
                   "l2": f"inputs larger than L2: {n_layers} layers' distinct caches of {cache_bytes / 1e6:.0f} MB "
                         f"and weights", "graph": "step replayed from a CUDA graph"},
        "kv_cache_gbs": n_layers * cache_bytes * steps_arg / (elapsed_ms / 1e3) / 1e9,
        "kv_bytes_per_token": (d.d_c + d.d_rope) * 2 + 4,
        "kv_bytes_per_token_model": n_layers // lgz * ((d.d_c + d.d_rope) * 2 + 4),
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                     "traffic": None, "kernel": "decode_tc_kernel", "kernel_ms": k_ms,
                     "bytes_per_launch": algo["total"], "bytes_breakdown": algo, "peak_source": peak_src},
        "projection_gemm": gemm,
        "cpu_baseline": cpu,
        "e2e": {"value": whole_job_rate(ws, B, e2e_steps, e2e_ms), "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h},
        # this library's kernels per layer: the query/latent projection,
        # kv_norm + RoPE, query absorption (with the append in its grid in the
        # first layer of a group), decode, the output projection
        "gpu_launches": steps_arg * n_layers * 5,
        "clocks": clk.summary(),
    }


def projection_gemm_timing(layers, torch, stream, peak, rounds=4):
    """The layer's two projection GEMMs alone (eg_mla_debug_linear on each
    layer's own weights and inputs, every layer in turn, so that the weights
    stream from HBM: 24 layers x 22 MB > L2): mean time per launch between
    CUDA events on the launching stream, and the weight bytes per launch over
    it (the batch rows and outputs are under 1 % of those bytes).  The launches
    run back to back from a captured graph, each allowed to start streaming
    its weights while the one before it finishes, as in the step."""
    from paper_2509_16686_gb300 import _lib
    res = {}
    for name in ("w_qkv_a", "w_o"):
        ops = []
        for layer in layers:
            w = getattr(layer, name)
            if name == "w_qkv_a":
                x, out = layer.x, torch.empty((layer.x.shape[0], w.shape[0]), dtype=torch.float32, device="cuda")
            else:
                u = layer.attn_output().reshape(layer.x.shape[0], -1)
                x, out = u, torch.empty((u.shape[0], w.shape[0]), dtype=torch.bfloat16, device="cuda")
            ops.append((w, x, out))
        with torch.cuda.stream(stream):
            for w, x, out in ops:
                _lib.eg_mla_debug_linear(w, x, out, stream=stream)
        stream.synchronize()
        # replayed from a captured graph, so that host launch costs drop out
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=stream):
            for w, x, out in ops:
                _lib.eg_mla_debug_linear(w, x, out, stream=stream)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            graph.replay()
            e0.record(stream)
            for _ in range(rounds):
                graph.replay()
            e1.record(stream)
        stream.synchronize()
        del graph
        ms = e0.elapsed_time(e1) / (rounds * len(ops))
        wbytes = ops[0][0].numel() * ops[0][0].element_size()
        gbs = wbytes / (ms * 1e-3) / 1e9
        res[name] = {"shape": [int(ops[0][0].shape[0]), int(ops[0][0].shape[1]), int(ops[0][1].shape[0])],
                     "kernel_ms": ms, "weight_bytes": wbytes, "achieved_gbs": gbs, "frac": gbs / peak}
    return res


def mla_baseline(case, torch, stream, peak, steps=600):
    """The same workload with the gate off (plain MLA over the same cached
    latents; the kernel's gate stage and the ids drop out): decode tokens/s of
    the step (graph over three cache replicas), the decode kernel's CUDA-event
    time, its roofline fraction and the cache bytes per token."""
    import dataclasses
    from paper_2509_16686_gb300 import _lib, device
    d = dataclasses.replace(case.dims, gate=False)
    mcase = dataclasses.replace(case, dims=d, name=case.name + "-mla")
    units = [device.upload(mcase) for _ in range(REPLICAS)]
    for r in units[1:]:
        for name in ("w_uk", "w_uv", "workspace", "status", "block_table"):
            setattr(r, name, getattr(units[0], name))
    with torch.cuda.stream(stream):
        for i in range(6):
            units[i % REPLICAS].step(stream)
    stream.synchronize()
    assert units[0].read_status() == 0, "device status (MLA baseline)"
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        for u in units:
            u.step(stream)
    reps = max(1, steps // REPLICAS)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        graph.replay()
        e0.record(stream)
        for _ in range(reps):
            graph.replay()
        e1.record(stream)
    torch.cuda.synchronize()
    ms_step = e0.elapsed_time(e1) / (reps * REPLICAS)
    _lib.eg_mla_profile_begin(3 * REPLICAS)
    pgraph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(pgraph, stream=stream):
        for _ in range(3):
            for u in units:
                u.step(stream)
    with torch.cuda.stream(stream):
        pgraph.replay()
        pgraph.replay()
    stream.synchronize()
    del pgraph
    ms_sum, n_l = _lib.eg_mla_profile_end()
    assert units[0].read_status() == 0, "device status (MLA baseline)"
    k_ms = ms_sum / max(1, n_l)
    tokens = int(case.seq_lens.astype(np.int64).sum())
    kvb = (d.d_c + d.d_rope) * (2 if d.dtype == "bf16" else 4)
    algo = algorithmic_bytes(mcase, tokens * kvb)
    achieved = algo["total"] / (k_ms * 1e-3) / 1e9
    del units, graph
    torch.cuda.empty_cache()
    return {"what": "the same workload with the gate off (plain MLA over the same latent cache)",
            "value": case.batch / (ms_step * 1e-3), "unit": UNIT, "ms_per_step": ms_step, "steps": reps * REPLICAS,
            "decode_kernel_ms": k_ms, "kv_bytes_per_token": kvb,
            "roofline": {"achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                         "bytes_per_launch": algo["total"], "bytes_breakdown": algo}}


def run_gpu_r0(args, workload, torch, dist, ws, rank):
    """The paper-literal (R0) gated decode, eg_mla_decode_r0, on the 4K-context
    shapes at batch 8 (d_c 256, vocabulary 32000): the up-projection of every
    cached row through W^UKV on tcgen05, the gate and LayerNorm over the 4096
    features of all heads, per-head attention.  Reported against the bf16
    tensor peak: the up-projection's FLOPs (2 x 4096 x d_c per cached token)
    over the whole call's time, a lower bound for the projection kernel."""
    from paper_2509_16686_gb300 import _lib, device, synth
    dev = torch.cuda.current_device()
    case = synth.case_c4k(batch=8, ctx=4096, keep_logical=False)
    r0 = synth.make_r0_inputs(case, seed=61)
    d = case.dims
    units = []
    for _ in range(REPLICAS):
        dc = device.upload(case)
        dc.append()
        units.append(dc)
    w_ukv = device.to_device_array(r0.w_ukv, "bf16", "cuda")
    gate = device.to_device_array(r0.gate_r0, "bf16", "cuda")
    gamma, beta = torch.from_numpy(r0.gamma).cuda(), torch.from_numpy(r0.beta).cuda()
    wsb = torch.empty(_lib.eg_mla_decode_r0_workspace_size(units[0].dims, case.batch, units[0].block_table.shape[1],
                                                           case.num_pages), dtype=torch.uint8,
                      device="cuda")
    out = torch.empty((case.batch, 16, 128), dtype=torch.bfloat16, device="cuda")
    stream = torch.cuda.Stream()

    def call(u):
        _lib.eg_mla_decode_r0(u.dims, u.q, u.c_pool, u.kr_pool, u.id_pool, u.block_table, u.seq_lens, w_ukv, gate,
                              gamma, beta, out, wsb, u.status, stream)

    with torch.cuda.stream(stream):
        for i in range(max(3, args.warmup)):
            call(units[i % REPLICAS])
    stream.synchronize()
    assert units[0].read_status() == 0, "device status (R0)"
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        for u in units:
            call(u)
    steps = args.steps if args.steps is not None else 60
    reps = max(1, steps // REPLICAS)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(nvsmi_id(torch, dev)) as clk:
        with torch.cuda.stream(stream):
            graph.replay()
            e0.record(stream)
            for _ in range(reps):
                graph.replay()
            e1.record(stream)
        torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / (reps * REPLICAS)
    assert units[0].read_status() == 0, "device status (R0)"
    tokens = int(case.seq_lens.astype(np.int64).sum())
    width = d.num_heads * (d.d_nope + d.d_v)
    flops = 2.0 * tokens * width * d.d_c
    peaks_path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(peaks_path):
        peak, src = float(json.load(open(peaks_path))["bf16_tflops"]), "measured"
    else:
        peak, src = 1900.0, "fallback"
    achieved = flops / (ms * 1e-3) / 1e12
    return {
        "metric": METRIC, "value": case.batch / (ms * 1e-3), "unit": UNIT, "n_gpus": ws,
        "steps": reps * REPLICAS, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": "r0: the paper-literal gate placement (gate and LayerNorm over the 4096 "
                               "up-projected key/value features of all heads), batch 8 x context 4096, 16 heads, "
                               "d_c 256, vocabulary 32000; seeded synthetic W^UKV (the case's W_UK, W_UV), "
                               "R0 gate table N(1, 0.1), gamma N(1, 0.1), beta N(0, 0.1)",
                   "batch": case.batch, "ctx_tokens_cached": tokens,
                   "l2": f"{REPLICAS} rotating cache replicas; the gated values of the pool "
                         f"({case.num_pages * 64 * d.num_heads * d.d_v * 2 / 1e6:.0f} MB) are written and read "
                         f"every step, and the R0 gate rows ({case.num_pages * 64 * width * 2 / 1e6:.0f} MB) read"},
        "roofline": {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                     "frac": achieved / peak, "traffic": None, "kernel": "r0_project_kernel (+ r0_attend_kernel)",
                     "flops_per_launch": flops, "peak_source": src,
                     "note": "up-projection FLOPs over the whole call (both kernels): a lower bound for the "
                             "projection kernel's tensor rate"},
        "gpu_launches": 2 * reps * REPLICAS,
        "clocks": clk.summary(),
    }


def prefill_case(workload):
    from paper_2509_16686_gb300 import synth
    if workload == "prefill":
        return synth.case_prefill(), ("prefill: 8 prompts x 4096 tokens, 16 heads, d_nope 128, d_rope 64, d_v 128, "
                                      "d_c 256, vocabulary 32000 (uniform ids), gate LN(c (*) G[id]), page 64")
    return synth.case_prefill_ragged(), ("prefill_ragged: 16 prompts of log-uniform lengths in [128, 4096], "
                                         "16 heads, d_c 192, vocabulary 50000, Zipf(1.1) ids, page 64")


def prefill_flops(pc):
    """Algorithmic FLOPs of one call: the causal attention (2 (d_n + d_r + d_v)
    per visible (query, key, head)) and the key/value up-projection
    (2 H (d_n + d_v) d_c per token)."""
    d = pc.dims
    pairs = sum(int(L) * (int(L) + 1) // 2 for L in pc.seq_lens)
    attn = 2.0 * pairs * d.num_heads * (d.d_nope + d.d_rope + d.d_v)
    proj = 2.0 * pc.total_tokens * d.num_heads * (d.d_nope + d.d_v) * d.d_c
    return attn, proj


def oracle_prefill_rate(pc, budget_s):
    """Prompt tokens/s of the fp64 oracle's prefill on host cores: whole heads
    of the first prompt while the budget lasts (at least one)."""
    from oracle import egmla_oracle as orc
    H = pc.dims.num_heads
    L = int(pc.seq_lens[0])
    t0 = time.perf_counter()
    done = 0
    for h in range(H):
        orc.prefill(pc, batches=[0], heads=[h])
        done += 1
        if time.perf_counter() - t0 > budget_s:
            break
    dt = time.perf_counter() - t0
    # prompt 0's tokens pass all H heads; the other prompts cost in proportion to L^2
    work_full = sum(int(x) ** 2 for x in pc.seq_lens) / float(L * L)
    rate = pc.total_tokens / (dt * H / done * work_full)
    return rate, (f"{done} of {H} heads of prompt 0 ({L} tokens), {dt:.1f} s, scaled by heads and by "
                  f"sum L^2 / L_0^2 = {work_full:.2f} to all prompts")


def run_gpu_prefill(args, workload, torch, dist, ws, rank):
    """Prompt processing through eg_mla_prefill (see the module docstring)."""
    from paper_2509_16686_gb300 import _lib, device
    dev = torch.cuda.current_device()
    pc, desc = prefill_case(workload)
    d = pc.dims
    dp = device.upload_prefill(pc)
    stream = torch.cuda.Stream()
    T = pc.total_tokens
    with torch.cuda.stream(stream):
        for _ in range(max(3, args.warmup)):
            dp.run(stream)
    stream.synchronize()
    assert dp.read_status() == 0, "device status (prefill)"
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        dp.run(stream)
    steps = args.steps if args.steps is not None else 200
    with torch.cuda.stream(stream):
        graph.replay()
    torch.cuda.synchronize()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(nvsmi_id(torch, dev)) as clk:
        if dist:
            dist.barrier()
        torch.cuda.synchronize()
        with torch.cuda.stream(stream):
            ev0.record(stream)
            for _ in range(steps):
                graph.replay()
            ev1.record(stream)
        torch.cuda.synchronize()
        if dist:
            dist.barrier()
    elapsed_ms = max_over_ranks(ev0.elapsed_time(ev1), dist, "cuda")
    assert dp.read_status() == 0, "device status (prefill)"
    ms = elapsed_ms / steps
    value = ws * T * steps / (elapsed_ms * 1e-3)

    # ---- the attention kernel alone: events around its launch in a captured
    # graph of 10 calls, replayed twice (the events hold the second replay)
    n_prof = 10
    _lib.eg_mla_profile_begin(n_prof)
    pgraph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(pgraph, stream=stream):
        for _ in range(n_prof):
            dp.run(stream)
    with torch.cuda.stream(stream):
        pgraph.replay()
        pgraph.replay()
    stream.synchronize()
    del pgraph
    ms_sum, n_l = _lib.eg_mla_profile_end()
    k_ms = ms_sum / max(1, n_l)
    attn_flops, proj_flops = prefill_flops(pc)
    peaks_path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(peaks_path):
        pk = json.load(open(peaks_path))
        peak, src = float(pk.get("bf16_tflops_sustained", pk["bf16_tflops"])), "measured (sustained)"
    else:
        peak, src = 1700.0, "fallback (sustained)"
    achieved = attn_flops / (k_ms * 1e-3) / 1e12

    # ---- end to end through the C ABI with host buffers: every step copies the
    # prompts' q, c, k^R and ids in from pinned host memory and reads the output back
    names = ("q", "c", "kr", "ids")
    h_in = {n: getattr(dp, n).cpu().pin_memory() for n in names}
    h_out = torch.empty(dp.out.shape, dtype=dp.out.dtype).pin_memory()
    h2d = sum(t.numel() * t.element_size() for t in h_in.values())
    d2h = h_out.numel() * h_out.element_size()
    e2e_steps = args.e2e_steps or min(steps, 50)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        e0.record(stream)
        for _ in range(e2e_steps):
            for n in names:
                getattr(dp, n).copy_(h_in[n], non_blocking=True)
            dp.run(stream)
            h_out.copy_(dp.out, non_blocking=True)
        e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1), dist, "cuda")
    e2e_value = ws * T * e2e_steps / (e2e_ms * 1e-3)
    assert dp.read_status() == 0, "device status (prefill e2e)"

    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        rate, sample = oracle_prefill_rate(pc, 12.0)
        cpu = {"value": rate, "unit": "tokens/s", "cores": BLAS_THREADS, "threads": BLAS_THREADS,
               "host_cores": host_cores(), "kind": "oracle", "sample": sample}
    return {
        "metric": "prefill tokens/sec (prompt tokens through gate, cache write, up-projection and causal attention)",
        "value": value, "unit": "tokens/s", "n_gpus": ws, "steps": steps, "warmup": args.warmup,
        "ms_per_step": ms, "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic",
        "config": {"workload": desc, "prompts": pc.batch, "tokens": T,
                   "l2": "inputs larger than L2 (q alone is "
                         f"{dp.q.numel() * 2 / 1e6:.0f} MB; the per-head keys and values "
                         f"{T * d.num_heads * 256 * 2 / 1e6:.0f} MB are rewritten every step)",
                   "graph": "one call per step, replayed from a CUDA graph"},
        "roofline": {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                     "frac": achieved / peak, "traffic": None, "kernel": "prefill_attn_kernel",
                     "kernel_ms": k_ms, "flops_per_launch": attn_flops, "peak_source": src,
                     "step_tflops": (attn_flops + proj_flops) / (ms * 1e-3) / 1e12,
                     "proj_flops_per_step": proj_flops},
        "cpu_baseline": cpu,
        "e2e": {"value": e2e_value, "unit": "tokens/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
        "gpu_launches": 3 * steps,
        "clocks": clk.summary(),
    }


def run_gpu(args, workload, torch, dist, ws, rank):
    """One bench line of `workload` (see the module docstring)."""
    if workload.startswith("prefill"):
        return run_gpu_prefill(args, workload, torch, dist, ws, rank)
    if workload == "r0":
        return run_gpu_r0(args, workload, torch, dist, ws, rank)
    if workload == "layers24_full":
        return run_gpu_full_layers(args, workload, torch, dist, ws, rank)
    from paper_2509_16686_gb300 import _lib, device  # noqa: F401
    dev = torch.cuda.current_device()
    case, desc = make_workload(workload)
    B = case.batch
    d = case.dims
    n_layers = layers_of(workload)
    steps_arg = args.steps if args.steps is not None else (200 if n_layers > 1 else
                                                          2000 if args.sweep else 20000)
    # units: one append + decode each.  A step runs one group of units: one of
    # REPLICAS rotating cache replicas (so consecutive steps stream different
    # memory), or all layers of the decoder.
    if n_layers > 1:
        base = device.upload(case, num_splits=args.splits)
        units = [base] + [device.clone_case(base) for _ in range(n_layers - 1)]
        groups = [units]
        l2_note = f"inputs larger than L2: {n_layers} layers' distinct caches"
    else:
        units = [device.upload(case, num_splits=args.splits) for _ in range(REPLICAS)]
        # replicas share the weights, block table and workspace of the first
        for r in units[1:]:
            for name in ("gate_table", "ln_gamma", "ln_beta", "w_uk", "w_uv", "workspace", "status",
                         "block_table"):
                setattr(r, name, getattr(units[0], name))
        groups = [[u] for u in units]
        l2_note = f"inputs larger than L2: {REPLICAS} rotating cache replicas"
    # each unit keeps its own per-step inputs, packed in one device buffer (one
    # host-to-device copy per unit in the end-to-end run), and its own output
    packed = [device.pack_step_inputs(u) for u in units]
    stream = torch.cuda.Stream()
    tokens_cached = int(case.seq_lens.astype(np.int64).sum())
    elem = 2 if d.dtype == "bf16" else 4
    id_bytes = 4 if d.gate else 0
    cache_bytes = tokens_cached * ((d.d_c + d.d_rope) * elem + id_bytes)     # per unit (layer)
    # algorithmic bytes of one decode launch: the cache stream, each distinct
    # gate row once, and W_UV of every head
    algo = algorithmic_bytes(case, cache_bytes)
    splits = units[0].num_splits or _lib.eg_mla_default_num_splits()
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    # bf16: query absorption (with the append in its grid) + decode, + the
    # combine kernel unless the decode kernel runs fused (d_c 192/256, a grid
    # of at most one CTA per SM); fp32: append + decode + combine
    fused = d.dtype == "bf16" and d.d_c in (192, 256) and splits <= sms
    launches_per_step = n_layers * ((2 if fused else 3) if d.dtype == "bf16" else 3)
    if workload.endswith("_embed"):
        launches_per_step += n_layers

    embed = workload.endswith("_embed")
    if embed:
        # the gate table of the step, computed in it from the embedding (the
        # units share the table tensor of the first)
        emb_h, w_ue_h = synth_mod().make_embedding(case, d.d_c, seed=75)
        emb_d = device.to_device_array(emb_h, "bf16", "cuda")
        w_ue_d = device.to_device_array(w_ue_h, "bf16", "cuda")

    def run_group(g):
        for u in g:
            if embed:
                _lib.eg_mla_gate_table(u.dims, emb_d, w_ue_d, u.gate_table, u.status, stream)
            u.step(stream)

    # ---- warm-up, then capture one graph of every group (one step each)
    with torch.cuda.stream(stream):
        for i in range(max(3, args.warmup)):
            run_group(groups[i % len(groups)])
    stream.synchronize()
    assert units[0].read_status() == 0, "device status after warm-up"
    # one graph of a step over every group in turn, replayed whole, and one
    # graph per group for the remainder, so that exactly `steps_arg` steps run
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        for g in groups:
            run_group(g)
    tail_graphs = []
    for g in groups[:steps_arg % len(groups)]:
        tg = torch.cuda.CUDAGraph()
        with torch.cuda.graph(tg, stream=stream):
            run_group(g)
        tail_graphs.append(tg)
    torch.cuda.synchronize()
    reps = steps_arg // len(groups)
    steps = reps * len(groups) + len(tail_graphs)
    with torch.cuda.stream(stream):
        for _ in range(2):
            graph.replay()
        for tg in tail_graphs:
            tg.replay()
    torch.cuda.synchronize()

    # ---- timed region: `steps` steps, barrier + sync on both sides
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(nvsmi_id(torch, dev)) as clk:
        if dist:
            dist.barrier()
        torch.cuda.synchronize()
        with torch.cuda.stream(stream):
            ev0.record(stream)
            for _ in range(reps):
                graph.replay()
            for tg in tail_graphs:
                tg.replay()
            ev1.record(stream)
        torch.cuda.synchronize()
        if dist:
            dist.barrier()
    elapsed_ms = max_over_ranks(ev0.elapsed_time(ev1), dist, "cuda")
    assert units[0].read_status() == 0, "device status after timed region"
    ms_per_step = elapsed_ms / steps
    value = whole_job_rate(ws, B, steps, elapsed_ms)

    # ---- the decode kernel alone: CUDA events around every decode launch,
    # recorded as nodes of a captured graph of the same steps (so that each
    # launch is timed as it runs in the step, without host launch gaps); the
    # graph is replayed twice and the events hold the second replay
    prof_groups = max(1, 10 // n_layers) * len(groups) if n_layers == 1 else 2
    _lib.eg_mla_profile_begin(prof_groups * len(groups[0]))
    pgraph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(pgraph, stream=stream):
        for i in range(prof_groups):
            run_group(groups[i % len(groups)])
    with torch.cuda.stream(stream):
        pgraph.replay()
        pgraph.replay()
    stream.synchronize()
    del pgraph
    ms_sum, n_l = _lib.eg_mla_profile_end()
    k_ms = ms_sum / max(1, n_l)
    achieved = algo["total"] / (k_ms * 1e-3) / 1e9
    peaks_path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(peaks_path):
        peak = float(json.load(open(peaks_path))["hbm_gbs"])
        peak_src = "measured"
    else:
        peak, peak_src = 6800.0, "fallback"
    traffic = None
    tpath = os.path.join(ROOT, "profiles", "traffic.json")
    if os.path.exists(tpath):
        tall = json.load(open(tpath))
        tj = tall.get(workload)
        if tj and tall.get("source_sha") == kernel_source_sha(tall.get("source_files", [])):
            traffic = tj.get("dram_bytes_per_launch")

    # ---- end to end through the C ABI with host buffers.  The units of the
    # steps run in order on the compute stream (each unit's two C calls bound
    # once, see _lib.bind_step); a copy stream carries the input copy of the
    # next unit (issued first, so it overlaps this one) and the read-back of
    # this unit's output.  Events order each unit's buffers between uses.
    e2e_steps = args.e2e_steps or min(steps, 2000 if n_layers == 1 else 100)
    pos = {id(u): k for k, u in enumerate(units)}
    seq = [pos[id(u)] for s_ in range(e2e_steps) for u in groups[s_ % len(groups)]]
    h_outs = [torch.empty(u.out.shape, dtype=u.out.dtype).pin_memory() for u in units]
    h2d = sum(packed[k][0].numel() * packed[k][0].element_size() for k in seq[:len(seq) // e2e_steps])
    d2h = sum(h_outs[k].numel() * h_outs[k].element_size() for k in seq[:len(seq) // e2e_steps])
    steps_bound = [u.bind(stream) for u in units]
    s_copy = torch.cuda.Stream()
    nu = len(units)
    ev_in = [torch.cuda.Event() for _ in units]
    ev_comp = [torch.cuda.Event() for _ in units]
    ev_out = [torch.cuda.Event() for _ in units]
    used = [False] * nu
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record(stream)
    s_copy.wait_stream(stream)
    with torch.cuda.stream(s_copy):
        packed[seq[0]][1].copy_(packed[seq[0]][0], non_blocking=True)
        ev_in[seq[0]].record(s_copy)
        for i, k in enumerate(seq):
            stream.wait_event(ev_in[k])
            if used[k]:
                stream.wait_event(ev_out[k])          # this unit's last output has been read back
            if embed:
                _lib.eg_mla_gate_table(units[k].dims, emb_d, w_ue_d, units[k].gate_table, units[k].status, stream)
            steps_bound[k]()
            ev_comp[k].record(stream)
            if i + 1 < len(seq):
                k1 = seq[i + 1]
                if used[k1] or k1 == k:
                    s_copy.wait_event(ev_comp[k1])    # the unit's last run has read its inputs
                packed[k1][1].copy_(packed[k1][0], non_blocking=True)
                ev_in[k1].record(s_copy)
            s_copy.wait_event(ev_comp[k])
            h_outs[k].copy_(units[k].out, non_blocking=True)
            ev_out[k].record(s_copy)
            used[k] = True
    stream.wait_stream(s_copy)
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1), dist, "cuda")
    e2e_value = whole_job_rate(ws, B, e2e_steps, e2e_ms)
    assert units[0].read_status() == 0, "device status after end-to-end run"

    # ---- the gate table from the embedding alone (c32k_embed): a graph of 20 calls
    gate_table = None
    if embed:
        gg = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gg, stream=stream):
            for _ in range(20):
                _lib.eg_mla_gate_table(units[0].dims, emb_d, w_ue_d, units[0].gate_table, units[0].status, stream)
        with torch.cuda.stream(stream):
            gg.replay()
            g0, g1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            g0.record(stream)
            gg.replay()
            g1.record(stream)
        torch.cuda.synchronize()
        gt_ms = g0.elapsed_time(g1) / 20
        V, d_e = case.dims.vocab, d.d_c
        gate_table = {"kernel": "prefill_kv_kernel (x W^T mode)", "ms": gt_ms, "vocab": V, "d_e": d_e,
                      "tflops": 2.0 * V * d_e * d.d_c / (gt_ms * 1e-3) / 1e12,
                      "bytes": (V * d_e + d.d_c * d_e + V * d.d_c) * 2,
                      "gbs": (V * d_e + d.d_c * d_e + V * d.d_c) * 2 / (gt_ms * 1e-3) / 1e9}
        del gg

    # ---- the gate-off (plain MLA) result of the same workload, beside the gated one
    mla = None
    if n_layers == 1 and d.gate and d.dtype == "bf16" and not args.no_mla_baseline and not args.sweep:
        mla = mla_baseline(case, torch, stream, peak)

    # ---- CPU baseline (rank 0, N = 1 only); a decode token passes every layer
    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline_line(case, 12.0, n_layers)

    return {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": steps, "warmup": args.warmup,
        "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": d.dtype, "data": "synthetic",
        "config": {"workload": desc, "batch": B, "layers": n_layers, "ctx_tokens_cached": tokens_cached,
                   "splits": splits, "page_size": d.page_size,
                   "l2": f"{l2_note} of {cache_bytes / 1e6:.0f} MB", "graph": "step replayed from a CUDA graph"},
        "kv_cache_gbs": n_layers * cache_bytes * steps / (elapsed_ms / 1e3) / 1e9,
        "kv_bytes_per_token": (d.d_c + d.d_rope) * elem + id_bytes,
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": traffic, "kernel": "decode_tc_kernel",
                     "kernel_ms": k_ms, "bytes_per_launch": algo["total"], "bytes_breakdown": algo,
                     "frac_cache_stream_only": cache_bytes / (k_ms * 1e-3) / 1e9 / peak,
                     "peak_source": peak_src},
        "cpu_baseline": cpu,
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
        "gpu_launches": steps * launches_per_step,
        "clocks": clk.summary(),
        "mla_baseline": mla,
        "gate_table": gate_table,
    }


def main():
    global LAYERS_OVERRIDE
    args = parse()
    if args.layers:
        LAYERS_OVERRIDE = args.layers
    if args.oracle_probe:
        return oracle_probe(args.oracle_probe, args.oracle_budget)
    if args.impl == "reference":
        return run_reference(args)
    import torch
    ws, rank, local = dist_env()
    dist = None
    if ws > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    workloads = [f"ctx{c}" for c in SWEEP_CTX] if args.sweep else [args.workload]
    for wl in workloads:
        line = run_gpu(args, wl, torch, dist, ws, rank)
        if rank == 0:
            print(json.dumps(line), flush=True)
        torch.cuda.empty_cache()
    if dist:
        dist.barrier()
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
