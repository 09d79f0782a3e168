"""Benchmark of one Chimera draft-and-verify step (7B-shaped model, batch 1).

A "step" is one pass of the whole hot path: K = 4 draft sub-steps (trigram encoder,
full-context block, residual head + top-k), tree expansion, the 64-node tree-masked
verify forward over 32 layers with the LM head and argmax, greedy acceptance, KV
compaction and the draft-KV append.  The model is random-init (N(0, 0.02)) with the
Vicuna-7B shape; the 512-token prompt is seeded uniform ids.

Output: one JSON line (rank 0).  `value` = tree tokens per second of whole steps (B * N
tree nodes per step, whole job); `ms_per_step` = device time of one step from CUDA
events around K back-to-back graph replays; `breakdown.verify_ms` = the verify phase
(tree expansion, 32-layer tree forward, LM head, argmax) from CUDA events recorded at
the phase boundaries of a graph replay; `e2e` = the same metric through chimera_step
with host output buffers and a synchronisation per step.  `--impl reference` times the
fp64 CPU oracle (whole steps on an oracle-prefilled state) instead.
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

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)
# the oracle's matrix products run on every host core
for _v in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
    os.environ.setdefault(_v, str(os.cpu_count() or 1))

import numpy  # noqa: E402,F401  (its BLAS starts with the thread count set above)
import torch  # noqa: E402

import synth  # noqa: E402

WORKLOAD = "7b"

# DRAM traffic of the dominant kernel (tensor-core linear or chain) over its
# algorithmic bytes (weights streamed once), from an ncu capture on a small case, keyed
# by the SHA-256 of the kernel source it was taken on: the roofline's `traffic` is
# null whenever the kernel has changed since (the key no longer matches).
LINEAR_TRAFFIC_RATIO = {
    # linear_tc.cu with red.global.add epilogues and two weight stages requested before
    # the dependency wait: dram__bytes_read.sum + dram__bytes_write.sum over weight
    # bytes, 3 launches each of 64 x 12288 x 4096 (1.053), 64 x 22016 x 4096 (1.054) and
    # 1 x 32000 x 8192 (1.003), weighted by the step's linear bytes (13.2 GB at 64 rows,
    # 4.3 GB at 1-5 rows)
    "8d9933dced1b9282721eb7136f71b4966e0a156fbbba06959cca43da6362f6e8": 1.041,
}


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def max_over_ranks(x: float, world: int) -> float:
    """The largest x over the ranks: a job's time is its slowest replica's."""
    if world <= 1:
        return x
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(units_per_rank: float, world: int, ms_job: float) -> float:
    """Units per second of the whole job: every replica processes units_per_rank in
    ms_job (the max over ranks)."""
    return world * units_per_rank / (ms_job * 1e-3)


def step_bytes(cfg, n_ctx):
    """Algorithmic HBM bytes of one step at committed lengths n_ctx (an int for batch 1,
    else one length per sequence).

    Every weight matrix counts once per use (the trigram encoder and the draft block
    once per draft sub-step, the heads once; a batch shares every weight read), embeddings
    only for the gathered rows, KV as the rows read at the model's element size (bf16: 2
    bytes per K or V value); the activations are excluded.  `kv_planes_extra` is what the
    stored hi + lo planes of precision mode 1 read on top (the same again): traffic, not
    algorithmic bytes."""
    d, F, V, L, K, N = (cfg["d_model"], cfg["ffn_dim"], cfg["vocab"], cfg["n_layers"],
                        cfg["n_draft_heads"], cfg["tree_nodes"])
    ns = [n_ctx] if isinstance(n_ctx, (int, float)) else list(n_ctx)
    B = len(ns)
    e = 2 if cfg["dtype"] == "bf16" else 4
    layer = (3 * d * d + d * d + 3 * d * F) * e
    kv_row = 2 * d * e
    verify_w = L * layer + V * d * e + B * N * d * e
    verify_kv = L * sum(n + N for n in ns) * kv_row
    draft_w = K * ((3 * d * d + d * d) * e + layer) + K * V * 2 * d * e + B * K * 3 * d * e
    draft_kv = sum((n + k + 1) * kv_row for n in ns for k in range(K))
    commit = 2 * d * d * e + B * 2 * L * 4 * kv_row
    return dict(verify=verify_w + verify_kv, verify_weights=verify_w, verify_kv=verify_kv,
                draft=draft_w + draft_kv, commit=commit, total=verify_w + verify_kv + draft_w + draft_kv + commit,
                kv_planes_extra=verify_kv + draft_kv)


WORKLOAD_NAMES = {
    "7b": "7B-shaped bs1 draft-and-verify step (N=64, topk 5,5,5,5, 512-token prompt)",
    "13b": "13B-shaped bs1 draft-and-verify step (N=64, topk 5,5,5,5, 2048-token prompt)",
    "7b_16k": "7B-shaped bs1 draft-and-verify step at a 16384-token context (N=64, paged KV block 16)",
    "7b_b8": "7B-shaped batch-8 ragged draft-and-verify step (N=32 per sequence, prompts 256..4096)",
}


def workload_config(cfg, prompt_len):
    return {"workload": WORKLOAD_NAMES[cfg["name"]],
            "batch": cfg["batch"], "tree_nodes": cfg["tree_nodes"], "prompt_len": prompt_len,
            "layers": cfg["n_layers"], "d_model": cfg["d_model"], "ffn_dim": cfg["ffn_dim"], "vocab": cfg["vocab"],
            "draft_heads": cfg["n_draft_heads"], "topk": cfg["topk"]}


def oracle_steps(cfg, w_cpu, prompt, n_steps, warmup=1):
    """The fp64 oracle (as it stands) on the host cores: prefill the prompt (setup,
    untimed), then `warmup` + n_steps whole draft-and-verify steps; returns the wall
    time of each timed step (s) and the setup time."""
    from oracle import chimera_oracle as co
    from oracle import tree as ot
    W = co.OracleWeights(w_cpu, cache=False)
    tree = ot.build_tree(cfg["topk"], cfg["tree_nodes"])
    cap = len(prompt) + (n_steps + warmup + 1) * 5 + cfg["tree_nodes"] + 8
    t0 = time.perf_counter()
    st = co.prefill(W, cfg, prompt, cap)
    setup = time.perf_counter() - t0
    for _ in range(warmup):
        co.step(W, cfg, st, tree)
    times = []
    for _ in range(n_steps):
        t0 = time.perf_counter()
        co.step(W, cfg, st, tree)
        times.append(time.perf_counter() - t0)
    return times, setup


def host_threads():
    try:
        aff = len(os.sched_getaffinity(0))
    except AttributeError:
        aff = os.cpu_count() or 1
    return {"cores": os.cpu_count() or 1, "affinity": aff, "blas_threads": int(os.environ["OPENBLAS_NUM_THREADS"])}


class Clocks:
    """nvidia-smi sampling during the timed region."""

    def __init__(self, index):
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
        try:
            self.p = subprocess.Popen(["nvidia-smi", f"--id={index}", f"--query-gpu={q}",
                                       "--format=csv,noheader,nounits", "-lms", "100"],
                                      stdout=self.f, stderr=subprocess.DEVNULL)
        except OSError:
            self.p = None

    def stop(self):
        if self.p is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.p.terminate()
        self.p.wait()
        self.f.flush()
        rows = [r.split(",") for r in open(self.f.name).read().strip().splitlines() if r.strip()]
        os.unlink(self.f.name)
        sm = [float(r[1]) for r in rows if len(r) >= 9 and r[1].strip().replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if len(r) >= 9 and r[2].strip().replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows if len(r) >= 9 for i in range(4)
                          if r[5 + i].strip().lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


def op_bench(args, hbm, peak_kind):
    """One kernel through its C-ABI entry point, on the operand shapes the 7B step
    launches, cycling through enough operand copies that every launch reads from HBM.
    This is the small case for per-kernel ncu captures (a few GB on the device)."""
    import paper_2402_15758_gb300 as pkg
    from paper_2402_15758_gb300 import build as pkg_build
    pkg_build.build()
    pkg.load()
    g = torch.Generator(device="cuda").manual_seed(0)
    dev = "cuda"
    if args.op == "linear":
        M, N, K = (int(v) for v in args.shape.split(","))
        wbytes = N * K * 2
        copies = max(2, -(-400_000_000 // wbytes))
        Ws = [(torch.randn(N, K, generator=g, device=dev) * 0.02).to(torch.bfloat16) for _ in range(copies)]
        X32 = torch.randn(M, K, generator=g, device=dev)
        X = X32.to(torch.bfloat16)
        X_lo = (X32 - X.float()).to(torch.bfloat16)
        # as in the step: fp32 output accumulated with red.add (the step zeroes it first)
        Y = torch.zeros(M, N, dtype=torch.float32, device=dev)
        nbytes = wbytes + 2 * M * K * 2 + M * N * 4

        def launch(i):
            pkg.op_linear(X, Ws[i % copies], Y, epi=2, out_f32=True, X_lo=X_lo, stream=stream)
        desc = (f"chimera_op_linear bf16 split operand (X_hi + X_lo), fp32 accumulate, M={M} N={N} K={K}, "
                f"{copies} weight copies ({copies * wbytes / 1e9:.2f} GB) cycled")
    else:
        H, hd, nq, n_ctx = 32, 128, 64, args.ctx
        n_keys = n_ctx + nq
        pages = (n_keys + 15) // 16
        lay = pages * H * 4 * 16 * hd * 2
        copies = max(2, -(-400_000_000 // lay))
        pools = [torch.randn(pages, H, 4, 16, hd, generator=g, device=dev).to(torch.bfloat16)
                 for _ in range(copies)]
        pt = torch.arange(pages, dtype=torch.int32, device=dev).reshape(1, pages)
        nctx = torch.tensor([n_ctx], dtype=torch.int32, device=dev)
        anc_l = []
        for i in range(nq):  # a 4-ary tree over the 64 rows: node i's parent is (i - 1) // 4
            m, j = 0, i
            while j >= 0:
                m |= 1 << j
                j = (j - 1) // 4 if j > 0 else -1
            anc_l.append(m - (1 << 64) if m >= 1 << 63 else m)
        anc = torch.tensor(anc_l, dtype=torch.int64, device=dev)
        q = torch.randn(nq, H * hd, generator=g, device=dev)
        out = torch.empty(nq, H * hd, dtype=torch.bfloat16, device=dev)
        out_lo = torch.empty_like(out)
        # as the step: one cluster of <= 8 CTAs per head, all heads resident at once
        splits = args.splits or max(1, min(8, torch.cuda.get_device_properties(0).multi_processor_count // H,
                                           -(-n_keys // 64)))
        nbytes = n_keys * H * hd * 4 * 2 + nq * H * hd * 4 + 2 * nq * H * hd * 2

        def launch(i):
            pkg.op_attention(q, pools[i % copies], pt, nctx, anc, out, nq=nq, q_local0=0, n_local=nq,
                             q_rows=nq, n_heads=H, head_dim=hd, splits=splits, out_lo=out_lo, stream=stream)
        desc = (f"chimera_op_attention 7B verify layer: 32 heads x 128, 64 tree rows, {n_ctx} context rows, "
                f"4 bf16 KV planes, {splits} KV splits, {copies} KV pools cycled")
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        for i in range(args.warmup):
            launch(i)
        stream.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        # the device sleeps while the host enqueues every launch, so the timed launches
        # run back to back (no host gaps inside the timed region)
        torch.cuda._sleep(int(2e6 * max(10, args.steps)))
        e0.record(stream)
        for i in range(args.steps):
            launch(i)
        e1.record(stream)
        stream.synchronize()
    ms = e0.elapsed_time(e1) / args.steps
    gbs = nbytes / (ms * 1e-3) / 1e9
    print(json.dumps({"op": args.op, "workload": desc, "us_per_launch": ms * 1e3, "bytes_per_launch": nbytes,
                      "achieved_gbs": gbs, "peak_gbs": hbm, "peak_kind": peak_kind, "frac": gbs / hbm,
                      "launches": args.steps, "note": "back-to-back device launches (enqueued behind a sleep kernel)"}))




def reference_arm(args, rank):
    """The oracle timed on the host cores, whole steps, on the main arm's workload."""
    if rank != 0:
        return
    cfg = synth.get_config(WORKLOAD)
    prompt = synth.make_prompts(cfg)[0]
    # the oracle reads the stored weights; draw them on the host with the same shapes
    w = synth.make_weights(cfg, device="cpu")
    ht = host_threads()
    times, setup = oracle_steps(cfg, w, prompt, args.steps, warmup=1)
    t = statistics.median(times)
    B, N = cfg["batch"], cfg["tree_nodes"]
    v = B * N / t
    sample = (f"whole steps of the fp64 NumPy oracle (draft K=4, 32-layer tree verify, LM head, accept, "
              f"commit) after an oracle prefill of the {len(prompt)}-token prompt ({setup:.1f} s, untimed); "
              f"1 warm-up + {args.steps} timed steps, median {t:.2f} s")
    line = {"impl": "reference", "metric": "tree tokens/s at 7B bs1 (draft-and-verify step)",
            "value": v, "unit": "tree tokens/s", "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": t * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": workload_config(cfg, len(prompt)),
            "cpu_baseline": {"kind": "oracle", "cores": ht["blas_threads"], "value": v, "unit": "tree tokens/s",
                             "sample": sample, "host": ht},
            "e2e": {"value": v, "unit": "tree tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "step_s": [round(x, 3) for x in times]}
    print(json.dumps(line))


def linear_traffic_ratio(kind):
    name = "chain_tc.cu" if kind == "chain" else "linear_tc.cu"
    src = os.path.join(ROOT, "paper_2402_15758_gb300", "csrc", name)
    h = hashlib.sha256(open(src, "rb").read()).hexdigest()
    return LINEAR_TRAFFIC_RATIO.get(h), h


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="chimera", choices=["chimera", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--layers", type=int, default=None,
                    help="profiling only: the 7B shapes with fewer base layers (not the benchmark workload)")
    ap.add_argument("--trigram-cache", type=int, default=0,
                    help="entries of the device trigram cache (0: off)")
    ap.add_argument("--fused-chain", action="store_true",
                    help="run the linears between two attentions as persistent chain launches (fused_chain = 1)")
    ap.add_argument("--workload", default=WORKLOAD, choices=sorted(WORKLOAD_NAMES),
                    help="the configuration stepped (default: the benchmark's, 7B bs1); the others are "
                         "measured the same way, without the CPU baseline")
    ap.add_argument("--op", choices=["linear", "attention"], default=None,
                    help="time one kernel entry point instead of the step")
    ap.add_argument("--shape", default="64,22016,4096", help="--op linear: M,N,K")
    ap.add_argument("--ctx", type=int, default=1024, help="--op attention: committed context rows")
    ap.add_argument("--splits", type=int, default=0, help="--op attention: KV splits per head (0: as the step)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.op:
        op_bench(args, *peaks())
        return
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        reference_arm(args, rank)
        return

    import paper_2402_15758_gb300 as pkg
    from paper_2402_15758_gb300 import build as pkg_build
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    torch.cuda.set_device(local)
    pkg_build.build()
    pkg.load()

    cfg = synth.get_config(args.workload)
    if args.layers:
        cfg["n_layers"] = args.layers
    if args.fused_chain:
        cfg["fused_chain"] = 1
    if args.trigram_cache:
        cfg["trigram_cache"] = args.trigram_cache
    B, N = cfg["batch"], cfg["tree_nodes"]
    prompts = synth.make_prompts(cfg)
    prompt = prompts[0]
    w = synth.make_weights(cfg, device="cuda")
    torch.cuda.synchronize()
    reps = max(3, min(args.steps, 20))
    total_steps = args.warmup + 3 * args.steps + reps + 8
    max_seq = ((max(len(p) for p in prompts) + total_steps * 5 + N + 64 + 15) // 16) * 16
    stream = torch.cuda.Stream()
    ctx = pkg.Chimera(cfg, w, max_batch=B, max_seq_len=max_seq, stream=stream)
    ctx.prefill(prompts)
    ctx.step_async(args.warmup)
    ctx.sync()
    n0s = [int(v) for v in ctx.read("n")[:B]]
    n0 = n0s[0]

    # ---- device-resident timing: K graph replays back to back ----
    clocks = Clocks(local)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.nvtx.range_push("timed_steps")
    e0.record(stream)
    ctx.step_async(args.steps)
    e1.record(stream)
    torch.cuda.nvtx.range_pop()
    ctx.sync()
    torch.cuda.synchronize()
    ms = max_over_ranks(e0.elapsed_time(e1) / args.steps, world)
    n1s = [int(v) for v in ctx.read("n")[:B]]
    n1 = n1s[0]
    mean_accept = sum(b - a for a, b in zip(n0s, n1s)) / (B * args.steps)

    # ---- per-step distribution: one event pair around each graph replay ----
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
    ev[0].record(stream)
    for i in range(args.steps):
        ctx.step_async(1)
        ev[i + 1].record(stream)
    ctx.sync()
    torch.cuda.synchronize()
    per_step = sorted(ev[i].elapsed_time(ev[i + 1]) for i in range(args.steps))

    def med_p90(xs):
        xs = sorted(xs)
        return statistics.median(xs), xs[min(len(xs) - 1, int(round(0.9 * (len(xs) - 1))))]

    step_median, step_p90 = (max_over_ranks(v, world) for v in med_p90(per_step))

    # ---- phases: events at the draft | verify | commit boundaries of a graph replay ----
    dr_ms, ve_ms, co_ms = ctx.profile_phases(args.steps)
    # the clocks were sampled through the timed replays and the two timing passes after
    # them (the timed region alone is shorter than the sampling interval)
    clk = clocks.stop()
    verify_med, verify_p90 = (max_over_ranks(v, world) for v in med_p90(ve_ms))
    draft_med, _ = med_p90(dr_ms)
    commit_med, _ = med_p90(co_ms)

    # ---- per-kernel timing, eager (an event pair around every launch: no overlap) ----
    rec = ctx.profile_step()
    launches = len(rec)
    kind_ms = {}
    for x in rec:
        kind_ms[x["kind"]] = kind_ms.get(x["kind"], 0.0) + x["ms"]
    # ---- the dominant kernel class alone: its launches of one step, back to back ----
    dom = max(("chain", "linear"), key=lambda k: kind_ms.get(k, 0.0))
    lin = ctx.profile_kind(dom, reps)
    att = ctx.profile_kind("attention", reps)

    # ---- end to end through chimera_step (host outputs, one sync per step) ----
    ctx.sync()
    if world > 1:
        torch.distributed.barrier()
    t0 = time.perf_counter()
    emitted = 0
    for _ in range(args.steps):
        out = ctx.step()
        emitted += sum(len(o) for o in out)
    t_e2e = max_over_ranks((time.perf_counter() - t0) / args.steps, world)
    hit_rate = None
    if args.trigram_cache:  # sub-steps whose trigram hit the cache, over a few more steps
        hits = []
        for _ in range(5):
            ctx.step()
            hits.append(float(ctx.read("trigram_hits").mean()))
        hit_rate = sum(hits) / len(hits)
    d2h = B * 4 + 4 + int(round(4 * emitted / args.steps))
    n_mid = [(a + b) // 2 for a, b in zip(n0s, n1s)]
    ctx.close()

    hbm, peak_kind = peaks()
    nb = step_bytes(cfg, n_mid)
    value = job_rate(B * N, world, ms)
    lin_per_launch_ms = lin["ms"] / max(1, lin["launches"])
    lin_bytes_per_launch = lin["bytes"] / max(1, lin["launches"])
    lin_gbs = lin_bytes_per_launch / (lin_per_launch_ms * 1e-3) / 1e9
    ratio, src_hash = linear_traffic_ratio(dom)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline and args.workload == WORKLOAD:
        w_cpu = {k: v.cpu() for k, v in w.items()}
        del w
        torch.cuda.empty_cache()
        ht = host_threads()
        times, setup = oracle_steps(cfg, w_cpu, prompt, 1, warmup=0)
        cpu = {"value": B * N / times[0], "unit": "tree tokens/s", "cores": ht["blas_threads"], "kind": "oracle",
               "sample": (f"one whole step of the fp64 NumPy oracle on its own prefilled state "
                          f"({len(prompt)}-token prompt, prefill {setup:.1f} s untimed): {times[0]:.2f} s"),
               "host": ht}
    line = {
        "metric": ("tree tokens/s at 7B bs1 (draft-and-verify step)" if args.workload == WORKLOAD
                   else f"tree tokens/s ({args.workload} draft-and-verify step)"),
        "value": value, "unit": "tree tokens/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": ms, "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic: random-init N(0,0.02) weights, uniform-random prompt ids",
        "config": dict(workload_config(cfg, [len(p) for p in prompts] if B > 1 else len(prompt)),
                       n_ctx=[n0s, n1s] if B > 1 else [n0, n1], parallelism="replicas" if world > 1 else "single",
                       precision="bf16 weights; split hi+lo bf16 GEMM operands, fp32 accumulation, "
                                 "KV cache as hi+lo bf16 planes",
                       l2=f"inputs larger than L2: {nb['total'] / 1e9:.1f} GB of weights and KV read per step"),
        "breakdown": {
            "verify_ms": verify_med, "verify_ms_p90": verify_p90, "draft_ms": draft_med, "commit_ms": commit_med,
            "phase_timing": "CUDA events at the phase boundaries of a graph replay of the step, one step at a time",
            "verify_tree_tokens_per_s": B * N / (verify_med * 1e-3),
            "step_ms_median": step_median, "step_ms_p90": step_p90,
            "step_bytes_gb": nb["total"] / 1e9, "verify_bytes_gb": nb["verify"] / 1e9,
            "kv_bytes_basis": "bf16 K and V values read (algorithmic); the hi+lo planes read "
                              f"{nb['kv_planes_extra'] / 1e9:.3f} GB more per step",
            "achieved_step_gbs": nb["total"] / (ms * 1e-3) / 1e9,
            "step_roofline_frac": nb["total"] / (ms * 1e-3) / 1e9 / hbm,
            "step_roofline_frac_8tbs": nb["total"] / (ms * 1e-3) / 1e9 / 8000.0,
            "verify_achieved_gbs": nb["verify"] / (verify_med * 1e-3) / 1e9,
            "verify_roofline_frac": nb["verify"] / (verify_med * 1e-3) / 1e9 / hbm,
            "verify_roofline_frac_8tbs": nb["verify"] / (verify_med * 1e-3) / 1e9 / 8000.0,
            "verify_roofline_ms": nb["verify"] / (hbm * 1e9) * 1e3,
            "attention_class_ms": att["ms"], "attention_launches": att["launches"],
            "kernel_ms_by_kind_eager": {k: round(v, 4) for k, v in sorted(kind_ms.items(), key=lambda t: -t[1])},
            "mean_accepted_tokens_per_step": mean_accept,
            "committed_tokens_per_s": B * mean_accept / (ms * 1e-3),
            "accept_note": "random-init draft heads: the draft rarely matches, so a step commits ~1 token "
                           "per sequence (the root); reported, not optimised",
        },
        "roofline": {"bound": "hbm",
                     "kernel": ("chain_kernel (persistent tcgen05 chain: the linears and row steps between two "
                                "attentions in one launch)") if dom == "chain" else
                               "tc_linear_kernel (tcgen05 weight-streaming linear)",
                     "achieved": lin_gbs, "peak": hbm, "peak_kind": peak_kind, "unit": "GB/s",
                     "frac": lin_gbs / hbm,
                     "traffic": (ratio * lin_bytes_per_launch) if ratio else None,
                     "traffic_basis": ("DRAM bytes per launch: small-case ncu ratio x algorithmic bytes"
                                       if ratio else f"no capture of this kernel source ({src_hash[:12]})"),
                     "bytes_per_launch": lin_bytes_per_launch, "ms_per_launch": lin_per_launch_ms,
                     "launches_per_step": lin["launches"], "ms_per_step": lin["ms"],
                     "timing": f"CUDA events around back-to-back replays of a graph holding only the step's "
                               f"{dom} launches (step order, programmatic dependent launch kept)"},
        "cpu_baseline": cpu,
        "e2e": {"value": job_rate(B * N, world, t_e2e * 1e3), "unit": "tree tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": d2h, "ms_per_step": t_e2e * 1e3},
        "gpu_launches": launches * args.steps,
        "clocks": clk,
    }
    if args.layers:
        line["config"]["workload"] += f" [profiling run: {args.layers} base layers, not the benchmark workload]"
    line["config"]["launch"] = "persistent chains" if args.fused_chain else "one launch per linear and row kernel"
    line["config"]["trigram_cache"] = args.trigram_cache
    if hit_rate is not None:
        line["breakdown"]["trigram_hit_rate"] = hit_rate
    if rank == 0:
        print(json.dumps(line))
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
