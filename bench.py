#!/usr/bin/env python
"""Benchmark of the GB300 repair path: repaired document tokens/s and p50 repair
latency per request, with the roofline fraction of the dominant kernel.

One step = one request through RepairSession.repair on one stream: the C-ABI
calls cr_assemble_compress (the encoder reading the chunk pool; for a bf16
cache the assembled copy is not written), cr_repair_forward and
cr_apply_residual_pool (the head reading the stale rows from the pool and
writing the repaired cache), captured once into a CUDA graph and replayed.
Default workload: the Llama-3.1-8B-shaped cache (32 layers, 8 KV heads,
head_dim 128, d_model 4096) with the d_c 512 / d_b 1024 / 6-block repairer,
one request of 10 chunks x 512 tokens.  Inputs are seeded and synthetic; the
pool (1 GiB) and the request's cache (0.67 GB, read from the pool and written
repaired) exceed the 129 MB L2, so no explicit L2 flush is needed between steps.

    python bench.py [--gpus N --steps K --warmup W] [--impl reference]
                    [--mask MODE] [--component kv|k|v] [--offset stale|zero]
                    [--keep-first-chunk] [--rope] [--train]

The last options time the attention-mask and output variants of App. F (and
the target's R_M on K) in place of the method's defaults; a variant run
names itself in config.variant and reports no e2e figure.  --train times one
AdamW update of the repair network per step instead (Sec. 4.2, App. A).

For N > 1 (torchrun, one process per GPU) every rank repairs its own request
stream with a weight replica: requests never interact, so there is no
collective; value = all ranks' tokens / the slowest rank's time.
`--impl reference` times the CPU oracle (float64 numpy) on a bounded prefix
of the same request instead.
"""
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

METRIC = "repaired doc tokens/s and p50 repair latency per request (1 GB300, % roofline)"
L2_BYTES = 129 * 1000 * 1000


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="llama8b")
    ap.add_argument("--chunks", type=int, default=None,
                    help="request of this many chunks instead of the workload's (same shapes; "
                         "a smaller case for profiling)")
    ap.add_argument("--no-graph", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--mask", default="block_causal",
                    choices=["block_causal", "token_causal", "bidirectional", "block_diagonal"])
    ap.add_argument("--component", default="kv", choices=["kv", "k", "v"])
    ap.add_argument("--offset", default="stale", choices=["stale", "zero"])
    ap.add_argument("--keep-first-chunk", action="store_true")
    ap.add_argument("--rope", action="store_true", help="apply the target's R_M to K after repair")
    ap.add_argument("--train", action="store_true",
                    help="time one training update (forward, objective, backward, AdamW) per step")
    args = ap.parse_args()
    args.variant = {k: v for k, v in (("mask", args.mask), ("component", args.component),
                                      ("offset", args.offset))
                    if v != {"mask": "block_causal", "component": "kv", "offset": "stale"}[k]}
    if args.keep_first_chunk:
        args.variant["keep_first_chunk"] = True
    if args.rope:
        args.variant["target_rope"] = True
    return args


def make_workload(F, args):
    if args.chunks is None:
        return F.make_case(args.workload)
    return F.make_case(args.workload, n_req_chunks=args.chunks, requests=None, batched=None)


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return p["hbm_gbs"], p["bf16_tflops"], p["bf16_tflops_sustained"], "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


def workload_desc(case):
    t, r = case.target, case.repairer
    lens = case.plan.request_lengths()
    nreq = len(lens)
    nch = len(case.plan.chunk_idx)
    return (f"{case.recipe.name}: target L{t.n_layers} H_kv{t.n_kv_heads} d_h{t.head_dim} "
            f"d_model{t.d_model} {t.cache_dtype}; repairer d_c{r.d_c} d_b{r.d_b} B{r.n_blocks} "
            f"{r.n_heads} heads MLP{r.mlp_hidden // r.d_b}x d_seg{r.d_seg}; {nreq} request(s), "
            f"{nch} chunks, {sum(lens)} tokens")


def sample_clocks(dev_index):
    """Start nvidia-smi sampling every 50 ms and wait (up to 10 s) for its first
    sample, so that the timed region that follows is covered."""
    path = tempfile.mktemp(prefix="cr_clocks_", suffix=".csv")
    q = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    try:
        f = open(path, "w")
        p = subprocess.Popen(["nvidia-smi", f"--query-gpu={q}", "--format=csv,noheader,nounits",
                              "-lms", "50", "-i", str(dev_index)], stdout=f,
                             stderr=subprocess.DEVNULL)
    except Exception:
        return None, None, path
    t0 = time.time()
    while time.time() - t0 < 10.0:
        f.flush()
        if os.path.getsize(path) > 0:
            break
        time.sleep(0.05)
    return p, f, path


def _smi_time(stamp):
    import datetime
    for fmt in ("%Y/%m/%d %H:%M:%S.%f", "%Y/%m/%d %H:%M:%S"):
        try:
            return datetime.datetime.strptime(stamp, fmt).timestamp()
        except ValueError:
            pass
    return None


def stop_clocks(handle, t_begin=None, t_end=None):
    """Samples taken between t_begin and t_end (host wall clock); all samples if
    none of them carries a usable timestamp."""
    p, f, path = handle
    if p is None:
        return None
    p.terminate()
    try:
        p.wait(timeout=5)
    except Exception:
        p.kill()
    f.close()
    rows = []
    with open(path) as fh:
        for line in fh:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) >= 10 and parts[2].replace(".", "").isdigit():
                rows.append(parts)
    os.unlink(path)
    if not rows:
        return None
    window, in_region = rows, False
    if t_begin is not None and t_end is not None:
        inside = [r for r in rows if (lambda ts: ts is not None and t_begin - 0.05 <= ts <= t_end + 0.05)(
            _smi_time(r[0]))]
        if inside:
            window, in_region = inside, True
    sm = [float(r[2]) for r in window]
    names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
    reasons = sorted({names[i] for r in window for i in range(4) if r[6 + i].lower() == "active"})
    pw = [float(r[4]) for r in window if r[4].replace(".", "").isdigit()]
    return {"sm_mhz": statistics.median(sm), "sm_max_mhz": float(window[0][3]),
            "power_w_max": max(pw) if pw else None, "reasons": reasons, "samples": len(window),
            "samples_in_timed_region": in_region}


def oracle_sample(case, n_chunks, max_tokens=None, mask="block_causal"):
    """Run the oracle on the first n_chunks of request 0 (a document prefix), cut to
    max_tokens tokens if given; returns (tokens, seconds)."""
    import numpy as np
    import oracle as O
    p = case.plan
    sel = p.chunk_idx[p.cu_chunks[0]:p.cu_chunks[1]][:n_chunks]
    kvs, embs = [], []
    for c in sel:
        kv, emb = case.pool_rows(int(p.chunk_start[c]), int(p.chunk_len[c]))
        kvs.append(kv)
        embs.append(emb)
    kv, emb = np.concatenate(kvs), np.concatenate(embs)
    lens = p.chunk_len[sel]
    cid = np.concatenate([np.full(l, i, np.int32) for i, l in enumerate(lens)])
    if max_tokens is not None and max_tokens < len(cid):
        kv, emb, cid = kv[:max_tokens], emb[:max_tokens], cid[:max_tokens]
    pos = np.arange(len(cid), dtype=np.int32)
    t, r = case.target, case.repairer
    t0 = time.perf_counter()
    O.repair_request(kv, emb, cid, pos, case.weights, cache_dtype=t.cache_dtype,
                     n_layers=t.n_layers, n_kv_heads=t.n_kv_heads, head_dim=t.head_dim,
                     n_heads=r.n_heads, mask_mode=mask)
    return len(cid), time.perf_counter() - t0


def max_over_ranks(ms, device):
    """The slowest rank's time: every rank of the process group passes its own and
    gets the maximum (no process group, or one rank: the value itself)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(ms)
    t = torch.tensor([float(ms)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(world, tokens_per_rank, steps, total_ms):
    """Weak scaling: every rank repairs its own tokens_per_rank per step; the rate is
    all ranks' tokens over the slowest rank's time."""
    return world * tokens_per_rank * steps / (total_ms / 1e3)


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    import fixtures as F
    case = make_workload(F, args)
    n_chunks = 1
    # each step repairs a prefix of the first chunk, sized so that the K timed
    # steps take about a minute of host time at any K
    cap = max(32, min(512, 25600 // max(args.steps, 1)))
    times, toks = [], 0
    for i in range(args.warmup + args.steps):
        n, s = oracle_sample(case, n_chunks, cap, args.mask)
        if i >= args.warmup:
            times.append(s)
            toks = n
    total = sum(times)
    value = toks * len(times) / total
    cores = os.cpu_count()
    sample = f"first {toks} tokens of the request's first chunk, full repair incl. head"
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * total / len(times), "p50_ms": 1e3 * statistics.median(times),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded), random-init repairer",
        "config": {"workload": workload_desc(case), "sample": sample},
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }))


def run_ours(args):
    import numpy as np
    import torch
    import torch.distributed as dist

    import fixtures as F
    from paper_2609_35139_gb300 import RepairSession, build, cr, dims_from, pack_host_weights

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    build.build()
    cr.lib()
    cr.cr_clear_device_status()

    case = make_workload(F, args)
    t, r = dims_from(case.target, case.repairer)
    pw = pack_host_weights(case.weights, case.repairer.n_blocks)
    p = case.plan
    kvp_h, embp_h = case.pool()
    to_dev = lambda a: (torch.from_numpy(a.view(np.int16)).view(torch.bfloat16)
                        if a.dtype == np.uint16 else torch.from_numpy(a)).cuda()
    kvp, embp = to_dev(kvp_h), to_dev(embp_h)
    N = p.n_tokens
    req_lens = p.request_lengths()
    sess = RepairSession(t, r, pw, max_tokens=N)
    stream = torch.cuda.current_stream()

    rope_mode = cr.CR_ROPE_GLOBAL if args.rope else cr.CR_ROPE_NONE
    freq = case.inv_freq_target if args.rope else None
    choice = dict(component=args.component, offset=args.offset, keep_first_chunk=args.keep_first_chunk)
    # RepairSession.repair's path: for a bf16 cache under the method's output the
    # encoder and the head read the pool, and no assembled cache is written
    pooled = (case.target.cache_dtype == "bf16" and args.component == "kv" and args.offset == "stale"
              and not args.keep_first_chunk)

    def head(f, mode):
        if pooled:
            sess.apply_pool(a, kvp, p.chunk_start, p.chunk_len, p.chunk_idx, p.cu_chunks, f, mode)
        else:
            sess.apply(a, f, mode, **choice)

    def step():
        sess.repair(kvp, embp, p.chunk_start, p.chunk_len, p.chunk_idx, p.cu_chunks, freq, rope_mode,
                    mask_mode=args.mask, **choice)

    # ---- per-call timing (eager), for the stage breakdown and the roofline
    a = sess.assemble(kvp, embp, p.chunk_start, p.chunk_len, p.chunk_idx, p.cu_chunks)
    # the step runs the fused front (assemble_compress) and the head as repair() does;
    # the two calls the front replaces are timed too, for the breakdown
    calls = [("assemble", lambda: sess.assemble(kvp, embp, p.chunk_start, p.chunk_len,
                                                p.chunk_idx, p.cu_chunks)),
             ("compress", lambda: sess.compress(a)),
             ("assemble_compress", lambda: sess.assemble_compress(kvp, embp, p.chunk_start,
                                                                  p.chunk_len, p.chunk_idx,
                                                                  p.cu_chunks, write_kv=not pooled)),
             ("forward", lambda: sess.forward(a, mask_mode=args.mask)),
             ("apply", lambda: head(freq, rope_mode))]
    for _ in range(3):
        for _, fn in calls:
            fn()
    torch.cuda.synchronize()
    stage_ms = {k: [] for k, _ in calls}
    for _ in range(10):
        for name, fn in calls:
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            fn()
            e1.record(stream)
            stage_ms[name].append((e0, e1))
    torch.cuda.synchronize()
    stages = {k: statistics.median(e0.elapsed_time(e1) for e0, e1 in v) for k, v in stage_ms.items()}

    # ---- the timed step: graph replay
    use_graph = not args.no_graph
    if use_graph:
        g = torch.cuda.CUDAGraph()
        step()
        torch.cuda.synchronize()
        with torch.cuda.graph(g):
            step()
        run = g.replay
    else:
        run = step
    for _ in range(args.warmup):
        run()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    # Inputs smaller than twice the L2 (129 MB): a 512 MB buffer is written between
    # steps, outside each step's events, so every step starts from a cold L2.
    es_c = 2 if case.target.cache_dtype == "bf16" else 4
    cache_bytes = N * case.target.d_kv * es_c
    flush = None
    if cache_bytes < 2 * L2_BYTES:
        flush = torch.empty(4 * L2_BYTES, dtype=torch.uint8, device="cuda")
    clk = sample_clocks(local)
    ev0 = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ev1 = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    t_begin = time.time()
    for i in range(args.steps):
        if flush is not None:
            flush.zero_()
        ev0[i].record(stream)
        run()
        ev1[i].record(stream)
    torch.cuda.synchronize()
    t_end = time.time()
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    clocks = stop_clocks(clk, t_begin, t_end)
    per_step = [ev0[i].elapsed_time(ev1[i]) for i in range(args.steps)]
    total_ms = max_over_ranks(sum(per_step), "cuda")
    value = whole_job_rate(world, N, args.steps, total_ms)
    l2_note = (f"L2 flushed between steps (512 MB written outside the timed events): the "
               f"request's cache ({cache_bytes / 1e6:.0f} MB) is under twice the 129 MB L2"
               if flush is not None else
               f"no flush: the request's cache ({cache_bytes / 1e6:.0f} MB) and the pool exceed the "
               f"129 MB L2")
    st, word = cr.cr_get_device_status()
    if st != cr.CR_OK:
        raise RuntimeError(f"device status {word}")

    # ---- end to end through the public API with host buffers
    e2e = None
    if not args.no_e2e and not args.variant:
        e2e = run_e2e(case, sess, kvp_h, embp_h, args, world)

    # ---- per-kernel rooflines; the one with the most time per step is reported
    hbm, tf_burst, tf_sus, src = load_peaks()
    tg, rp = case.target, case.repairer
    es = 2 if tg.cache_dtype == "bf16" else 4
    head_cols = tg.d_kv if args.component == "kv" else tg.d_kv // 2
    head_flops = 2.0 * N * rp.d_b * head_cols
    # cr_apply_residual is one kernel launch (a V-only choice under R_M adds the K rotation)
    head_ms = stages["apply"]
    attn_flops, attn_ms = attention_timing(case, sess, a, args.mask)
    # The method applies the target's R_M to K after the repair (Sec. 4.1); the step
    # above leaves K canonical. The head with R_M, timed like the other calls (after
    # the timed region, so that the launch order before it is unchanged).
    if not args.rope and not args.variant:
        fn = lambda: head(case.inv_freq_target, cr.CR_ROPE_GLOBAL)
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        ev = []
        for _ in range(10):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            fn()
            e1.record(stream)
            ev.append((e0, e1))
        torch.cuda.synchronize()
        stages["apply_rope"] = statistics.median(e0.elapsed_time(e1) for e0, e1 in ev)
    gather_bytes = 2.0 * N * (tg.d_kv + tg.d_model) * es
    # the fused front's HBM work: the pool's cache rows read (and, without the pool
    # head, the assembled copy written), the embeddings read and written
    front_bytes = N * (tg.d_kv + 2 * tg.d_model) * es if pooled else gather_bytes
    kernels = {
        "attn_kernel": dict(name=f"attn_kernel ({args.mask.replace('_', '-')} flash attention)",
                            launches=rp.n_blocks,
                            ms=attn_ms, flops=attn_flops,
                            algorithmic=f"4*d_b per visible (query, key) pair = {attn_flops:.3e} "
                                        f"flop per launch"),
        "gemm_kernel<256,KV>": dict(name=("cr_apply_residual_pool" if pooled else "cr_apply_residual")
                                    + " (KV residual head GEMM + residual add)",
                                    launches=1, ms=head_ms, flops=head_flops,
                                    algorithmic=f"2*N*d_b*(columns visited) = {head_flops:.3e} "
                                                f"flop per launch"),
    }
    dom_key = max(kernels, key=lambda k: kernels[k]["launches"] * kernels[k]["ms"])
    dom = kernels[dom_key]
    achieved = dom["flops"] / (dom["ms"] * 1e-3) / 1e12
    # the kernel is timed in isolated calls (ten eager launches, CUDA events): the
    # burst peak applies
    roofline = {"kernel": dom["name"], "bound": "tensor", "achieved": achieved, "peak": tf_burst,
                "unit": "TFLOP/s", "frac": achieved / tf_burst,
                # DRAM counters were taken on the method's workload, not on a variant
                "traffic": None if args.variant else traffic_from_profiles(dom_key),
                "peak_source": f"{src} bf16_tflops (burst: the kernel timed in isolated calls)",
                "algorithmic": dom["algorithmic"], "launch_ms": dom["ms"],
                "launches_per_step": dom["launches"]}
    # Whole request: the algorithmic tensor work at the sustained bf16 peak (the step
    # loop keeps the tensor cores busy through the whole timed region) plus the
    # front's HBM work (the pool read; the assembled write where the head does not
    # read the pool) at the measured copy bandwidth; the segment projection's flops
    # ride on that traffic.
    S = 2 * tg.n_layers * tg.n_kv_heads
    lin_flops = 2.0 * N * (S * rp.d_seg * rp.d_c + tg.d_model * rp.d_c + 2 * rp.d_c * rp.d_b
                           + rp.n_blocks * rp.d_c * rp.d_b
                           + rp.n_blocks * (4 * rp.d_b * rp.d_b + 2 * rp.d_b * rp.mlp_hidden))
    enc_flops = 2.0 * N * (S * rp.d_seg * rp.d_c + tg.d_model * rp.d_c + 2 * rp.d_c * rp.d_b
                           + rp.n_blocks * rp.d_c * rp.d_b)
    tensor_flops = lin_flops + rp.n_blocks * attn_flops + head_flops
    ideal_ms = tensor_flops / (tf_sus * 1e12) * 1e3 + front_bytes / (hbm * 1e9) * 1e3
    roofline.update({
        "request_frac": ideal_ms / (total_ms / args.steps),
        "request_frac_p50": ideal_ms / statistics.median(per_step),
        "request_ideal_ms": ideal_ms,
        "request_algorithmic": (f"{tensor_flops:.4e} tensor flop (linears {lin_flops:.3e}, attention "
                                f"{rp.n_blocks * attn_flops:.3e}, head {head_flops:.3e}) at the sustained "
                                f"{tf_sus} TF/s + {front_bytes:.4e} front bytes at {hbm} GB/s"),
    })
    stage_roofline = {
        "assemble_hbm_frac": gather_bytes / (stages["assemble"] * 1e-3) / 1e9 / hbm,
        "assemble_hbm_gbs": gather_bytes / (stages["assemble"] * 1e-3) / 1e9,
        # fused front: its cache and embedding bytes plus the encoder's small GEMMs,
        # over the whole call
        "front_hbm_frac": front_bytes / (stages["assemble_compress"] * 1e-3) / 1e9 / hbm,
        # the front against its own floor: its HBM bytes at the copy bandwidth plus the
        # encoder's algorithmic flops (W_map, P_tok, F, P_b) at the burst peak
        "front_frac": (front_bytes / (hbm * 1e9) + enc_flops / (tf_burst * 1e12)) * 1e3 /
                      stages["assemble_compress"],
        "front_ms": stages["assemble_compress"],
        "attention_tensor_frac": attn_flops / (attn_ms * 1e-3) / 1e12 / tf_burst,
        "attention_ms_per_launch": attn_ms,
        "head_tensor_frac": head_flops / (head_ms * 1e-3) / 1e12 / tf_burst,
        "peaks": f"{src}: HBM {hbm} GB/s, bf16 {tf_burst} TF/s burst for isolated kernels",
        "head_ms": head_ms,
    }
    if "apply_rope" in stages:
        stage_roofline["head_rope_tensor_frac"] = head_flops / (stages["apply_rope"] * 1e-3) / 1e12 / tf_burst
        stage_roofline["head_rope_ms"] = stages["apply_rope"]
    # front: gather (embeddings + chunk map), sigma fold, projection, the encoder's
    # GEMMs (W_map with P_tok and F with P_b as two-product launches where d_c and
    # d_b are whole 256-column tiles, else one launch each) and the two-term split
    # of s|e (fp32 caches: the two-call path with its two bf16 conversions);
    # forward: RoPE table, 7 kernels per block, final LayerNorm; head (with the pool
    # head, the pool-row table first)
    enc = (1 if rp.d_c % 256 == 0 else 2) + \
        ((1 if rp.d_b % 256 == 0 else 2) if rp.n_blocks > 0 else 1)
    launches_per_step = 1 + 2 + enc + 1 + (2 if tg.cache_dtype == "f32" else 0) \
        + (1 if rp.n_blocks > 0 else 0) + 7 * rp.n_blocks + 1 + 1 + (1 if pooled else 0)
    launches_per_step += 1 if (args.mask == "block_diagonal" and rp.n_blocks > 0) else 0
    launches_per_step += 1 if (args.rope and args.component == "v") else 0
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        # the whole first request: about 10-30 s of oracle work on the host cores
        n_chunks = int(case.plan.cu_chunks[1] - case.plan.cu_chunks[0])
        ntok, secs = oracle_sample(case, n_chunks, mask=args.mask)
        cpu = {"value": ntok / secs, "unit": "tokens/s", "cores": os.cpu_count(), "kind": "oracle",
               "sample": f"first {n_chunks} chunks ({ntok} tokens) of the request, full repair "
                         f"incl. head, float64 numpy, {secs:.1f} s"}
    if rank == 0:
        out = {
            "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": total_ms / args.steps,
            "p50_ms": statistics.median(per_step),
            "p90_ms": sorted(per_step)[int(0.9 * (len(per_step) - 1))],
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (seeded caches, embeddings, chunk map; random-init Xavier repairer)",
            "config": {"workload": workload_desc(case), "n_tokens": N, "cuda_graph": use_graph,
                       "n_requests": len(req_lens),
                       "request_tokens": {"min": min(req_lens), "mean": sum(req_lens) / len(req_lens),
                                          "max": max(req_lens)},
                       "latency": ("one call repairs every request of the step; each request is "
                                   "complete when the call is, so p50 is each request's latency"
                                   if len(req_lens) > 1 else "one request per step"),
                       "l2": l2_note,
                       "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
                       **({"variant": args.variant} if args.variant else {})},
            "roofline": roofline, "stage_roofline": stage_roofline,
            "stages_ms": stages, "cpu_baseline": cpu, "e2e": e2e,
            "gpu_launches": launches_per_step * args.steps, "clocks": clocks,
        }
        print(json.dumps(out))
    if world > 1:
        dist.destroy_process_group()


def attention_timing(case, sess, a, mask="block_causal", iters=10):
    """Per-launch time of the attention kernel at this workload's shapes (same chunk
    map, mask and launch configuration as inside the forward) and its algorithmic
    flops: 4 d_b per visible (query, key) pair."""
    import numpy as np
    import torch
    from paper_2609_35139_gb300 import cr
    rp = case.repairer
    N = a.n_tokens
    qkv = torch.randn(N, 3 * rp.d_b, device="cuda").to(torch.bfloat16)
    out = torch.empty(N, rp.d_b, device="cuda", dtype=torch.bfloat16)
    starts = torch.empty(N, dtype=torch.int32, device="cuda")
    cr.cr_chunk_starts(sess.chunk_end, a.cu_seqlens, N, starts)
    run = lambda: cr.cr_masked_attention(qkv, rp.d_b, rp.n_heads, mask, sess.chunk_end, starts,
                                         a.cu_seqlens, out)
    for _ in range(3):
        run()
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(iters):
        run()
    e1.record(stream)
    torch.cuda.synchronize()
    cend = sess.chunk_end[:N].to(torch.int64).cpu().numpy()
    cstart = starts[:N].to(torch.int64).cpu().numpy()
    cu = np.asarray(a.cu_seqlens, np.int64)
    local = np.arange(N) - np.repeat(cu[:-1], np.diff(cu))
    lens = np.repeat(np.diff(cu), np.diff(cu))
    visible = {"block_causal": cend, "token_causal": local + 1, "bidirectional": lens,
               "block_diagonal": cend - cstart}[mask]
    return 4.0 * rp.d_b * float(visible.sum()), e0.elapsed_time(e1) / iters


def traffic_from_profiles(kernel_key):
    """DRAM bytes per launch from a committed ncu summary, if it was taken on the
    kernel source as it is now (else None)."""
    import hashlib
    import re
    files = {"attn_kernel": ("attention_llama8b.md", "cr_attn.cu"),
             "gemm_kernel<256,KV>": ("head_gemm_llama8b.md", "cr_gemm.cu")}
    if kernel_key not in files:
        return None
    prof, srcf = files[kernel_key]
    try:
        with open(os.path.join(ROOT, "profiles", prof)) as f:
            text = f.read()
        with open(os.path.join(ROOT, "paper_2609_35139_gb300", "csrc", srcf), "rb") as f:
            sha = hashlib.sha256(f.read()).hexdigest()
    except OSError:
        return None
    m = re.search(r"traffic_bytes_per_launch:\s*(\d+)", text)
    h = re.search(r"source_sha256:\s*([0-9a-f]{64})", text)
    if not m or not h or h.group(1) != sha:
        return None
    return int(m.group(1))


def run_e2e(case, sess, kvp_h, embp_h, args, world):
    """Through the public serving API (RepairPipeline): every step copies the
    request's chunk caches from a pinned host pool to the device, repairs them and
    copies the repaired cache back to pinned host memory.  The pipeline overlaps a
    step's transfers with the neighbouring steps' repairs (two slots, copy streams
    in both directions); the timed region starts from an idle device and ends when
    the last repaired cache is in host memory."""
    import numpy as np
    import torch
    from paper_2609_35139_gb300 import RepairPipeline

    p = case.plan
    sel = p.chunk_idx[p.cu_chunks[0]:p.cu_chunks[1]]
    lens = p.chunk_len[sel]
    starts = p.chunk_start[sel]
    pin = lambda a: (torch.from_numpy(a.view(np.int16)).view(torch.bfloat16)
                     if a.dtype == np.uint16 else torch.from_numpy(a)).pin_memory()
    kv_h, emb_h = pin(kvp_h), pin(embp_h)
    N = int(lens.sum())
    pipe = RepairPipeline(sess.target, sess.rep, sess.weights, max_tokens=N)
    outs = [torch.empty(N, kv_h.shape[1], dtype=kv_h.dtype).pin_memory() for _ in range(2)]

    def run(k):
        for i in range(k):
            pipe.submit(kv_h, emb_h, starts, lens, outs[i % 2])
        pipe.drain()

    run(args.warmup)
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream()
    # three timed batches of K requests, the median reported: the host link is
    # shared with the machine's other GPUs and one batch can catch a burst of
    # their traffic
    batches = []
    for _ in range(3):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        run(args.steps)
        e1.record(stream)
        torch.cuda.synchronize()
        batches.append(e0.elapsed_time(e1) / args.steps)
    ms = statistics.median(batches)
    es = kv_h.element_size()
    return {"value": world * N / (ms / 1e3), "unit": "tokens/s", "ms_per_step": ms,
            "h2d_bytes_per_step": int(N * (kv_h.shape[1] + emb_h.shape[1]) * es),
            "d2h_bytes_per_step": int(N * kv_h.shape[1] * es),
            "batches_ms_per_step": batches,
            "path": "RepairPipeline: pinned host chunks -> device staging (H2D stream) -> three "
                    "C-ABI calls (compute stream: fused assembly + encoder, repair blocks, head) "
                    "-> pinned host repaired cache (D2H stream); "
                    "two slots, transfers overlapped with the neighbouring requests' repairs"}


def train_flops(case, visible_pairs):
    """Algorithmic flops of one update: the forward's linears, head, segment projection and
    attention (visible pairs only), and the backward's two products per linear (dX, dW; the
    segment projection needs dW only), the FC1 recompute and 2.5x the attention's work
    (S again, dV, dP, dQ, dK against S and PV forward)."""
    t, r = case.target, case.repairer
    N = case.plan.n_tokens
    S = 2 * t.n_layers * t.n_kv_heads
    dc, db, B, hid = r.d_c, r.d_b, r.n_blocks, r.mlp_hidden
    lin = 2.0 * N * (S * r.d_seg * dc + t.d_model * dc + 2 * dc * db + B * dc * db
                     + B * (4 * db * db + 2 * hid * db))
    head = 2.0 * N * db * t.d_kv
    seg = 2.0 * N * t.d_kv * r.d_seg
    attn = B * 4.0 * db * visible_pairs
    return 3 * lin + 3 * head + 2 * seg + 2.0 * N * db * hid * B + 3.5 * attn


def run_train(args):
    """One AdamW update of the repair network per step (Sec. 4.2, App. A) on the
    workload's request against a seeded synthetic joint cache (stale + sigma_Delta noise),
    through cr_train_step: eager launches, every kernel the library's own."""
    import numpy as np
    import torch

    import fixtures as F
    from paper_2609_35139_gb300 import RepairSession, TrainSession, build, cr, dims_from, pack_host_weights

    if int(os.environ.get("WORLD_SIZE", "1")) > 1:
        raise SystemExit("--train runs on one GPU: data-parallel training would need a gradient "
                         "all-reduce, which is not built")
    torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
    build.build()
    cr.lib()
    cr.cr_clear_device_status()
    case = make_workload(F, args)
    t, r = dims_from(case.target, case.repairer)
    p = case.plan
    kvp_h, embp_h = case.pool()
    to_dev = lambda a: (torch.from_numpy(a.view(np.int16)).view(torch.bfloat16)
                        if a.dtype == np.uint16 else torch.from_numpy(a)).cuda()
    N = p.n_tokens
    sess = RepairSession(t, r, pack_host_weights(case.weights, case.repairer.n_blocks), max_tokens=N)
    a = sess.assemble(to_dev(kvp_h), to_dev(embp_h), p.chunk_start, p.chunk_len, p.chunk_idx, p.cu_chunks)
    kv = sess.kv[:N]
    g = torch.Generator(device="cuda").manual_seed(7)
    sd = torch.from_numpy(case.weights["sigma_delta"]).cuda()
    joint = (kv.float() + sd[None] * torch.randn(kv.shape, device="cuda", generator=g)).to(torch.bfloat16)
    lens = np.diff(a.cu_seqlens)
    ts = TrainSession(t, r, case.weights, N, int(lens.max()))
    del sess.h0, sess.rein, sess.yf, sess.workspace
    step = lambda: ts.step(kv, joint, sess.emb[:N], sess.chunk_end[:N], sess.pos[:N], a.cu_seqlens, N, 3e-4,
                           mask_mode=args.mask)
    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    loss0 = float(ts.stats[0].item())
    stream = torch.cuda.current_stream()
    clk = sample_clocks(int(os.environ.get("LOCAL_RANK", "0")))
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
    t_begin = time.time()
    evs[0].record(stream)
    for i in range(args.steps):
        step()
        evs[i + 1].record(stream)
    torch.cuda.synchronize()
    t_end = time.time()
    clocks = stop_clocks(clk, t_begin, t_end)
    per = [evs[i].elapsed_time(evs[i + 1]) for i in range(args.steps)]
    total_ms = evs[0].elapsed_time(evs[-1])
    st, word = cr.cr_get_device_status()
    if st != cr.CR_OK:
        raise RuntimeError(f"device status {word}")
    cend = sess.chunk_end[:N].to(torch.int64).cpu().numpy()
    cid = sess.chunk_id[:N].to(torch.int64).cpu().numpy()
    local = np.arange(N) - np.repeat(a.cu_seqlens[:-1], lens)
    starts = np.array([np.searchsorted(cid[a.cu_seqlens[q]:a.cu_seqlens[q + 1]], cid[t], "left")
                       for q in range(len(lens)) for t in range(a.cu_seqlens[q], a.cu_seqlens[q + 1])])
    visible = {"block_causal": cend, "token_causal": local + 1, "bidirectional": np.repeat(lens, lens),
               "block_diagonal": cend - starts}[args.mask]
    flops = train_flops(case, float(visible.sum()))
    hbm, tf_burst, tf_sus, src = load_peaks()
    achieved = flops / (total_ms / args.steps * 1e-3) / 1e12
    B = case.repairer.n_blocks
    # launches per update (all of them this library's kernels): forward 10 + 7 B,
    # objective 5 (row weights, the loss head, row sums, request sums, total), head
    # backward 6, 28 per block backward (10 of them the tcgen05 dW / dX products; bias
    # sums fused with the bf16 conversion), encoder backward 12, clipping and AdamW 3
    launches = 36 + 35 * B if B > 0 else 0
    print(json.dumps({
        "metric": "trained doc tokens/s (one AdamW update of the repair network per step, 1 GB300)",
        "value": N * args.steps / (total_ms / 1e3), "unit": "tokens/s", "n_gpus": 1,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": total_ms / args.steps,
        "p50_ms": statistics.median(per), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16 GEMM operands, fp32 accumulation and master weights",
        "data": "synthetic (seeded caches, embeddings, joint = stale + sigma_Delta noise; random-init repairer)",
        "config": {"workload": workload_desc(case), "n_tokens": N, "variant": {"train": True, **args.variant},
                   "l2": "no flush: the cache, joint cache and residual buffers exceed L2",
                   "optimizer": "AdamW (0.9, 0.95), wd 0.01, clip 1.0, lr 3e-4"},
        "roofline": {"kernel": "whole update (forward, objective, backward, AdamW)", "bound": "tensor",
                     "achieved": achieved, "peak": tf_sus, "unit": "TFLOP/s", "frac": achieved / tf_sus,
                     "traffic": None, "algorithmic": f"{flops:.3e} flop per update",
                     "peak_source": f"{src} bf16_tflops_sustained"},
        "loss_first_timed": loss0, "loss_last": float(ts.stats[0].item()),
        "gpu_launches": launches * args.steps, "clocks": clocks,
    }))


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
    elif args.train:
        run_train(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
