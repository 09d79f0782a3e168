"""Benchmark of one Chimera draft-and-verify step (7B-shaped model, batch 1).

A "step" is one pass of the whole hot path: K = 4 draft sub-steps (trigram encoder,
full-context block, residual head + top-k), tree expansion, the 64-node tree-masked
verify forward over 32 layers with the LM head and argmax, greedy acceptance, KV
compaction and the draft-KV append.  The model is random-init (N(0, 0.02)) with the
Vicuna-7B shape; the 512-token prompt is seeded uniform ids.

Output: one JSON line (rank 0).  `value` = tree tokens per second (B * N tree nodes
verified per step, whole job); `ms_per_step` = device time of one step from CUDA
events around K back-to-back graph replays; `e2e` = the same metric through
chimera_step with host output buffers and a synchronisation per step.
`--impl reference` times the fp64 CPU oracle instead (see `cpu_sample`).
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

import synth  # noqa: E402

WORKLOAD = "7b"
LINEAR_DRAM_BYTES_PER_STEP = 18.23e9


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


def step_bytes(cfg, n_ctx, kv_elem_bytes=None):
    """Algorithmic HBM bytes of one step at committed length n_ctx (batch 1).

    Every weight matrix counts once per use (the trigram encoder and the draft block
    once per draft sub-step), embeddings only for the gathered rows, KV as the rows
    read; activations are excluded.  kv_elem_bytes is the stored size of one K (or V)
    element: 4 for the fp32-equivalent hi+lo bf16 planes of precision mode 1, else the
    weight element size."""
    d, F, V, L, K, N = (cfg["d_model"], cfg["ffn_dim"], cfg["vocab"], cfg["n_layers"],
                        cfg["n_draft_heads"], cfg["tree_nodes"])
    e = 2 if cfg["dtype"] == "bf16" else 4
    layer = (3 * d * d + d * d + 3 * d * F) * e
    kv_row = 2 * d * (kv_elem_bytes or e)
    verify = L * layer + V * d * e + N * d * e + L * (n_ctx + N) * kv_row
    draft_w = K * ((3 * d * d + d * d) * e + layer) + K * V * 2 * d * e + K * 3 * d * e
    draft_kv = sum((n_ctx + k + 1) * kv_row for k in range(K))
    commit = 2 * d * d * e + 2 * L * 4 * kv_row
    return dict(verify=verify, draft=draft_w + draft_kv, commit=commit,
                total=verify + draft_w + draft_kv + commit)


class Clocks:
    """nvidia-smi sampling during the timed region."""

    def __init__(self, index):
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
        try:
            self.p = subprocess.Popen(["nvidia-smi", f"--id={index}", f"--query-gpu={q}",
                                       "--format=csv,noheader,nounits", "-lms", "200"],
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


def cpu_sample(cfg, w_dev, n_ctx, threads):
    """Time the fp64 oracle on host cores on a bounded sample of the step:
    one base layer of the tree verify (64 nodes, n_ctx committed rows), the LM head on
    64 rows, and one draft sub-step (trigram encoder, full-context block row, one head).
    The step estimate scales the layer by the layer count and the draft sub-step by K."""
    from oracle import chimera_oracle as co
    from oracle import tree as ot
    names = ["embed", "lm_head", "final_norm", "tri_w1", "tri_w2", "heads.0"]
    names += [n for n in w_dev if n.startswith("layers.0.") or n.startswith("draft.")]
    w = {n: w_dev[n].cpu() for n in names}
    W = co.OracleWeights(w, cache=False)
    H, hd, d, N = cfg["n_heads"], cfg["head_dim"], cfg["d_model"], cfg["tree_nodes"]
    rng = np.random.default_rng(0)
    tree = ot.build_tree(cfg["topk"], N)
    mask = np.array([[(tree["anc"][i] >> j) & 1 == 1 for j in range(N)] for i in range(N)])
    ctx_k = rng.standard_normal((n_ctx, H, hd))
    ctx_v = rng.standard_normal((n_ctx, H, hd))
    x = rng.standard_normal((N, d))
    pos = n_ctx + np.array(tree["depth"])
    t0 = time.perf_counter()
    out, _, _ = co.block_rows(W, "layers.0", cfg, x, pos, ctx_k, ctx_v, mask)
    t_layer = time.perf_counter() - t0
    t0 = time.perf_counter()
    hs = co.rmsnorm(out, W("final_norm"), cfg["rms_eps"])
    _ = hs @ W("lm_head").T
    t_lm = time.perf_counter() - t0
    t0 = time.perf_counter()
    t = co.trigram_input(W, cfg, [1, 2, 3])
    g = co.trigram_encoder(W, t)
    h, _, _ = co.block_rows(W, "draft", cfg, g[None], np.array([n_ctx]), ctx_k, ctx_v, np.ones((1, 1), bool))
    z = W("heads.0") @ np.concatenate([hs[0], h[0]])
    _ = co.topk_desc(z, max(cfg["topk"]))
    t_draft = time.perf_counter() - t0
    est = cfg["n_layers"] * t_layer + t_lm + cfg["n_draft_heads"] * t_draft
    return dict(t_layer=t_layer, t_lm=t_lm, t_draft_sub=t_draft, step_s=est, threads=threads)


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
        splits = max(1, min(8, torch.cuda.get_device_properties(0).multi_processor_count // H, -(-n_keys // 64)))
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


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="chimera", choices=["chimera", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--profile-steps", type=int, default=3)
    ap.add_argument("--op", choices=["linear", "attention"], default=None,
                    help="time one kernel entry point instead of the step")
    ap.add_argument("--shape", default="64,22016,4096", help="--op linear: M,N,K")
    ap.add_argument("--ctx", type=int, default=1024, help="--op attention: committed context rows")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.op:
        op_bench(args, *peaks())
        return

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    cfg = synth.get_config(WORKLOAD)
    B, N = cfg["batch"], cfg["tree_nodes"]
    prompt = synth.make_prompts(cfg)[0]
    threads = os.cpu_count() or 1

    if args.impl == "reference":
        if rank != 0:
            return
        torch.manual_seed(0)
        # the oracle needs only the weights of the sampled parts; draw them on the host
        # with the same shapes (values do not change the timing)
        w = synth.make_weights(dict(cfg, n_layers=1), device="cpu")
        for _ in range(args.warmup if args.warmup < 1 else 1):
            cpu_sample(cfg, w, len(prompt), threads)
        times = [cpu_sample(cfg, w, len(prompt), threads)["step_s"] for _ in range(args.steps)]
        t = statistics.median(times)
        v = B * N / t
        line = {"impl": "reference", "metric": "tree tokens/s at 7B bs1 (draft-and-verify step)",
                "value": v, "unit": "tree tokens/s", "n_gpus": args.gpus, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": t * 1e3, "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
                "config": {"workload": "7B-shaped bs1 draft-and-verify step (N=64, topk 5,5,5,5, 512-token prompt)"},
                "cpu_baseline": {"kind": "oracle", "cores": threads, "value": v, "unit": "tree tokens/s",
                                 "sample": "per step: one verify layer (64 nodes, 512 ctx) x32 + LM head + "
                                           "one draft sub-step x4, fp64 NumPy on the host cores"},
                "e2e": {"value": v, "unit": "tree tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
        print(json.dumps(line))
        return

    import paper_2402_15758_gb300 as pkg
    from paper_2402_15758_gb300 import build as pkg_build
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    torch.cuda.set_device(local)
    pkg_build.build()
    pkg.load()

    w = synth.make_weights(cfg, device="cuda")
    torch.cuda.synchronize()
    total_steps = args.warmup + 2 * args.steps + args.profile_steps + args.steps + 8
    max_seq = ((len(prompt) + total_steps * 5 + N + 64 + 15) // 16) * 16
    stream = torch.cuda.Stream()
    ctx = pkg.Chimera(cfg, w, max_batch=B, max_seq_len=max_seq, stream=stream)
    ctx.prefill([prompt])
    ctx.step_async(args.warmup)
    ctx.sync()
    n0 = int(ctx.read("n")[0])

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
    clk = clocks.stop()
    n1 = int(ctx.read("n")[0])
    mean_accept = (n1 - n0) / args.steps

    # ---- per-step distribution: one event pair around each graph replay ----
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
    ev[0].record(stream)
    for i in range(args.steps):
        ctx.step_async(1)
        ev[i + 1].record(stream)
    ctx.sync()
    torch.cuda.synchronize()
    per_step = sorted(ev[i].elapsed_time(ev[i + 1]) for i in range(args.steps))
    step_median = max_over_ranks(statistics.median(per_step), world)
    step_p90 = max_over_ranks(per_step[min(len(per_step) - 1, int(round(0.9 * (len(per_step) - 1))))], world)

    # ---- per-kernel timing (eager launches with events around each) ----
    recs = []
    for _ in range(args.profile_steps):
        recs.append(ctx.profile_step())
    launches = len(recs[-1])

    def agg(pred):
        out = []
        for r in recs:
            sel = [x for x in r if pred(x)]
            out.append((sum(x["ms"] for x in sel), sum(x["bytes"] for x in sel), len(sel)))
        return out

    lin = agg(lambda x: x["kind"] == "linear")
    lin_ms = statistics.median([a[0] for a in lin])
    lin_bytes = statistics.median([a[1] for a in lin])
    lin_n = lin[-1][2]
    phase_ms = {ph: statistics.median([a[0] for a in agg(lambda x, ph=ph: x["phase"] == ph)])
                for ph in ("draft", "verify", "commit")}
    eager_ms = statistics.median([sum(x["ms"] for x in r) for r in recs])
    kind_ms = {}
    for x in recs[-1]:
        kind_ms[x["kind"]] = kind_ms.get(x["kind"], 0.0) + x["ms"]

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
    d2h = B * 4 + 4 + int(round(4 * emitted / args.steps))

    hbm, peak_kind = peaks()
    nb = step_bytes(cfg, (n0 + n1) // 2, kv_elem_bytes=4 if ctx.kv_f32 else None)
    value = job_rate(B * N, world, ms)
    if lin_ms <= 0:
        raise RuntimeError("per-kernel profile returned no linear time")
    lin_gbs = lin_bytes / (lin_ms * 1e-3) / 1e9
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cs = cpu_sample(cfg, w, n1, threads)
        cpu = {"value": B * N / cs["step_s"], "unit": "tree tokens/s", "cores": threads, "kind": "oracle",
               "sample": (f"fp64 NumPy oracle: one verify layer (64 nodes, {n1} ctx) {cs['t_layer']:.2f}s x32 + "
                          f"LM head {cs['t_lm']:.2f}s + one draft sub-step {cs['t_draft_sub']:.2f}s x4 "
                          f"= {cs['step_s']:.1f}s per step (estimate)")}
    line = {
        "metric": "tree tokens/s at 7B bs1 (draft-and-verify step)",
        "value": value, "unit": "tree tokens/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": ms, "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic: random-init N(0,0.02) weights, uniform-random prompt ids",
        "config": {"workload": "7B-shaped bs1 draft-and-verify step (N=64, topk 5,5,5,5, 512-token prompt)",
                   "batch": B, "tree_nodes": N, "prompt_len": len(prompt), "n_ctx": [n0, n1],
                   "parallelism": "replicas" if world > 1 else "single",
                   "precision": "bf16 weights; split hi+lo bf16 GEMM operands, fp32 accumulation, "
                                "KV cache as hi+lo bf16 planes (fp32-equivalent)",
                   "l2": "inputs larger than L2: 17.8 GB of weights streamed per step"},
        "breakdown": {
            "verify_ms_eager": phase_ms["verify"], "draft_ms_eager": phase_ms["draft"],
            "commit_ms_eager": phase_ms["commit"], "step_ms_eager": eager_ms,
            "step_ms_median": step_median, "step_ms_p90": step_p90,
            "kernel_ms_by_kind": {k: round(v, 4) for k, v in sorted(kind_ms.items(), key=lambda t: -t[1])},
            "step_bytes_gb": nb["total"] / 1e9, "verify_bytes_gb": nb["verify"] / 1e9,
            "achieved_step_gbs": nb["total"] / (ms * 1e-3) / 1e9,
            "step_roofline_frac": nb["total"] / (ms * 1e-3) / 1e9 / hbm,
            "step_roofline_frac_8tbs": nb["total"] / (ms * 1e-3) / 1e9 / 8000.0,
            "verify_roofline_frac_eager": nb["verify"] / (phase_ms["verify"] * 1e-3) / 1e9 / hbm,
            "mean_accepted_tokens_per_step": mean_accept,
        },
        "roofline": {"bound": "hbm", "kernel": "linear_tc (tcgen05 weight-streaming linear)",
                     "achieved": lin_gbs, "peak": hbm, "peak_kind": peak_kind, "unit": "GB/s",
                     "frac": lin_gbs / hbm, "traffic": LINEAR_DRAM_BYTES_PER_STEP,
                     "traffic_basis": "DRAM bytes read + written by all linear launches of one step (ncu)",
                     "launches_per_step": lin_n, "bytes_per_step": lin_bytes, "ms_per_step": lin_ms},
        "cpu_baseline": cpu,
        "e2e": {"value": job_rate(B * N, world, t_e2e * 1e3), "unit": "tree tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": d2h, "ms_per_step": t_e2e * 1e3},
        "gpu_launches": launches * args.steps,
        "clocks": clk,
    }
    ctx.close()
    if rank == 0:
        print(json.dumps(line))
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
