"""Benchmark of the DAS-Wave hot path on GB300.

One step = one pass of the whole hot path over one batch of synthetic input:
  draft   L Mature-V draft-attention calls (keys at depth r, values at R),
  verify  L full-depth verify-attention calls (depth R) over w candidate rows,
  accept  greedy acceptance over [B, w, vocab] fp32 logits,
  append  commit of the accepted inputs' K/V at all R depths and L layers.
The default workload is long-context drafting (B4 L4 H32/8 D128 P32768 T16,
R = 32, r = 6) on its full cache layout: all 32 depth slabs of K and V
allocated (68.8 GB), keys read at depth r and values at depth R.
`value` is the Mature-V draft attention's prefix-KV bandwidth (GB/s): the
algorithmic bytes the draft calls must read (K at depth r plus V at depth R,
sum_b P_b * Hkv * D * 2 bytes each, per layer) over their device time,
measured with CUDA events on the launch stream.  Inputs are resident in HBM
before the timed region; L2 is flushed before every timed step (a 512 MiB
buffer written, then read back so that no dirty line of it is left for the
timed region to write back).  `e2e` repeats the draft phase through the
public Python/C API with the step's inputs copied from pinned host memory
and its outputs read back.  The other workloads' attention phases, greedy
acceptance and the commit at the verify-and-commit shape, sequential
drafting, a DAS-Wave refinement and the e4m3 cache variant are reported as
extra keys, each timed the same way.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
    python bench.py --impl reference ...   # the fp64 CPU oracle on host cores

With N > 1 (torchrun) every rank runs an independent replica on its own GPU
(the path has no exchange step); value = bytes of all ranks / max time.
"""
import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

DEFAULT_WORKLOAD = "long"
FALLBACK_HBM_GBS = 6800.0


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3000)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="das", choices=["das", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-probes", action="store_true",
                    help="skip the long-prefix draft-phase measurements")
    ap.add_argument("--layers", type=int, default=0,
                    help="override the workload's layer count (smaller profiling captures)")
    ap.add_argument("--probe", default="",
                    help="run only one probe (draft:<workload>, e4m3:decode, e4m3:long, "
                         "commit:verify) with --steps/--warmup/--layers and print its result: "
                         "for profiling captures")
    ap.add_argument("--compact-depths", action="store_true",
                    help="store 2 depths (key depth 1, value depth 2) instead of R: the same "
                         "bytes per call in a smaller cache, for profiling captures")
    ap.add_argument("--clock-ms", type=int, default=20,
                    help="nvidia-smi sampling interval during the timed region")
    return ap.parse_args()


def flush_l2(buf):
    """Evict L2 before a timed step.  The buffer (four times the 129 MB L2) is
    written, then read back: the read makes L2 write the dirty lines back to
    HBM before the timed region, which otherwise pays for up to 129 MB of
    write-backs as its first loads evict them.  What stays in L2 is clean
    lines of this buffer, which no timed kernel reads."""
    buf.fill_(1)
    buf.sum()


def max_over_ranks(values, world, device):
    """Each timing value as the maximum over the ranks (the slowest replica
    sets the whole job's time); the values of this rank when world == 1."""
    import torch
    import torch.distributed as dist

    t = torch.tensor(list(values), dtype=torch.float64, device=device)
    if world > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return t.tolist()


def whole_job_gbs(world, bytes_per_step, steps, seconds):
    """Whole-job throughput: the bytes all ranks processed (each rank a full
    replica of the workload) over the slowest rank's time."""
    return world * bytes_per_step * steps / seconds / 1e9


def dist_env():
    return (int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)),
            int(os.environ.get("LOCAL_RANK", 0)))


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, "fallback"


def graph_kernel_nodes(graph):
    """Kernel nodes of a captured torch CUDA graph, read with the driver API
    (cuGraphGetNodes, cuGraphNodeGetType); None if either is unavailable."""
    import ctypes
    raw = getattr(graph, "raw_cuda_graph", None)
    if raw is None:
        return None
    try:
        cu = ctypes.CDLL("libcuda.so.1")
    except OSError:
        return None
    h = ctypes.c_void_p(raw())
    n = ctypes.c_size_t(0)
    if cu.cuGraphGetNodes(h, None, ctypes.byref(n)) != 0:
        return None
    nodes = (ctypes.c_void_p * max(1, n.value))()
    if cu.cuGraphGetNodes(h, nodes, ctypes.byref(n)) != 0:
        return None
    kind, kernels = ctypes.c_int(0), 0
    for i in range(n.value):
        if cu.cuGraphNodeGetType(ctypes.c_void_p(nodes[i]), ctypes.byref(kind)) != 0:
            return None
        kernels += kind.value == 0  # CU_GRAPH_NODE_TYPE_KERNEL
    return kernels


def code_digest(path):
    """code_text_digest of a source file."""
    return code_text_digest(open(path, encoding="utf-8").read())


def code_text_digest(text):
    """First 16 hex digits of the sha256 of a C/C++/CUDA source with its
    comments, trailing blanks and empty lines removed (string and character
    literals kept), so that an edit of comments alone keeps the digest."""
    out, i, n = [], 0, len(text)
    while i < n:
        c = text[i]
        if c in "\"'":
            j = i + 1
            while j < n and text[j] != c:
                j += 2 if text[j] == "\\" else 1
            out.append(text[i:j + 1])
            i = j + 1
        elif text.startswith("//", i):
            j = text.find("\n", i)
            i = n if j < 0 else j
        elif text.startswith("/*", i):
            j = text.find("*/", i + 2)
            i = n if j < 0 else j + 2
        else:
            out.append(c)
            i += 1
    code = "\n".join(line.rstrip() for line in "".join(out).splitlines() if line.strip())
    return hashlib.sha256(code.encode()).hexdigest()[:16]


def kernel_traffic(workload):
    """dram bytes per attention launch from the committed ncu summary, if the
    kernel's code has not changed since it was captured; else None."""
    src = os.path.join(ROOT, "paper_2609_34538_gb300", "csrc", "das_attention.cu")
    digest = code_digest(src)
    path = os.path.join(ROOT, "profiles", "attn_kernel_traffic.txt")
    if not os.path.exists(path):
        return None
    for line in open(path):
        parts = line.split()
        if len(parts) == 3 and parts[0] == workload and parts[1] == digest:
            return float(parts[2])
    return None


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons while running."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index, interval_ms=20):
        self.index = index
        self.interval_ms = interval_ms
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", str(self.interval_ms)],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            # wait for the first sample so that the timed region is covered
            self.first = self.proc.stdout.readline()
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *exc):
        self.lines = []
        if self.proc is not None:
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                out, _ = self.proc.communicate()
            # samples taken while the timed region ran (the first one came before)
            self.lines = [l for l in out.splitlines() if l.strip()]

    def summary(self):
        if not getattr(self, "lines", None):
            return None
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for l in self.lines:
            f = [x.strip() for x in l.split(",")]
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except (ValueError, IndexError):
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ----------------------------------------------------------------------------- GPU arm

def gpu_arm(args):
    import torch
    import torch.distributed as dist

    import paper_2609_34538_gb300 as das
    from synth import device as sdev
    from synth import workloads as wlm

    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    dev = torch.device("cuda", local)
    if args.probe:  # one probe alone (profiling captures); no benchmark line
        kind, _, name = args.probe.partition(":")
        fn = {"draft": draft_probe, "e4m3": f8_probe, "commit": commit_probe}.get(kind)
        if fn is None or name not in wlm.WORKLOADS:
            raise SystemExit(f"bench: unknown probe {args.probe!r}")
        peak, _ = peaks()
        kw = {"compact": args.compact_depths} if kind == "draft" else {}
        print(json.dumps({"probe": args.probe, **fn(name, dev, args.steps, args.warmup, peak,
                                                     layers=args.layers, **kw)}))
        return
    wl = wlm.WORKLOADS[args.workload]
    if args.layers:
        wl = wl.replace(layers=args.layers)
    if args.compact_depths:
        wl = wl.replace(depths=2, key_depth=1, value_depth=2)
    if wl.kind != "draft":
        raise SystemExit("the benchmark step needs a draft workload (its verify pass is derived)")
    R, L, B = wl.depths, wl.layers, wl.batch
    W = wl.max_block            # verify width: the draft block's rows are the candidates
    vocab = 32000
    wlv = wl.replace(key_depth=R, value_depth=R, seed=wl.seed + 1)

    stream = torch.cuda.Stream(device=dev)
    with torch.cuda.stream(stream):
        K, V = sdev.build_cache(wl, key_depths={wl.key_depth, R}, value_depths={R}, device=dev)
        cache = das.DepthKVCache(K, V)
        P0 = torch.from_numpy(wl.prefix_lens()).to(dev)
        pl = P0.clone()
        bl = torch.from_numpy(wl.block_lens()).to(dev)
        ws = das.new_workspace(cache, wl.q_heads, W, device=dev)
        draft_in = [sdev.layer_inputs(wl, l, dev) for l in range(L)]
        verify_in = [sdev.layer_inputs(wlv, l, dev) for l in range(L)]
        outs = [(torch.empty_like(q), torch.empty((B, wl.q_heads, W), dtype=torch.float32,
                                                  device=dev)) for q, _, _ in draft_in]
        vouts = [(torch.empty_like(q), torch.empty((B, wl.q_heads, W), dtype=torch.float32,
                                                   device=dev)) for q, _, _ in verify_in]
        acc_wl = wl.replace(vocab=vocab)
        a_star, draft_ids, logits = sdev.accept_tensors(acc_wl, dev)
        accepted = torch.empty(B, dtype=torch.int32, device=dev)
        target = torch.empty((B, W), dtype=torch.int32, device=dev)
        nxt = torch.empty(B, dtype=torch.int32, device=dev)
        kn, vn = sdev.build_staged(wl, W, device=dev)
        flag = torch.zeros(1, dtype=torch.int32, device=dev)
        flush = torch.empty(512 * 2 ** 20, dtype=torch.uint8, device=dev)
    stream.synchronize()

    def draft_phase():
        for l, (q, kb, vb) in enumerate(draft_in):
            das.das_mature_v_attention(cache, l, wl.key_depth, wl.value_depth, pl, bl, q, kb, vb,
                                       ws, out=outs[l][0], lse=outs[l][1], stream=stream)

    def verify_phase():
        for l, (q, kb, vb) in enumerate(verify_in):
            das.das_verify_attention(cache, l, R, pl, bl, q, kb, vb, ws, out=vouts[l][0],
                                     lse=vouts[l][1], stream=stream)

    def commit_phase():
        das.das_greedy_accept(logits, draft_ids, accepted, target, nxt, stream=stream)
        das.das_kv_append(cache, kn, vn, accepted, pl, flag, stream=stream)

    # one eager pass (library set-up), then CUDA graphs of the three phases
    with torch.cuda.stream(stream):
        pl.copy_(P0)
        draft_phase(); verify_phase(); commit_phase()
    stream.synchronize()
    # the library's launches per step: the kernel nodes of the three graphs
    # (each holds library calls only), read before they are instantiated;
    # the count of the launch sequence (L attention + L merge per attention
    # phase, accept 1 or 2, append 2) if the graph cannot be read
    graphs, nodes = [], []
    for fn in (draft_phase, verify_phase, commit_phase):
        try:
            g = torch.cuda.CUDAGraph(keep_graph=True)
        except TypeError:
            g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            fn()
        try:
            nodes.append(graph_kernel_nodes(g))
        except RuntimeError:
            nodes.append(None)
        if hasattr(g, "instantiate"):
            g.instantiate()
        graphs.append(g)
    launches_per_step = (sum(nodes) if None not in nodes else None)

    def step(ev):
        with torch.cuda.stream(stream):
            pl.copy_(P0)          # every step commits onto the same prefix
            flush_l2(flush)       # evict L2 (129 MB) before the timed phases
            ev[0].record(stream)
            graphs[0].replay()
            ev[1].record(stream)
            graphs[1].replay()
            ev[2].record(stream)
            graphs[2].replay()
            ev[3].record(stream)

    mk = lambda: [torch.cuda.Event(enable_timing=True) for _ in range(4)]
    for _ in range(args.warmup):
        step(mk())
    stream.synchronize()
    evs = [mk() for _ in range(args.steps)]
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local, args.clock_ms) as clocks:
        t0 = time.perf_counter()
        for e in evs:
            step(e)
        torch.cuda.synchronize()
        wall = time.perf_counter() - t0
    if world > 1:
        dist.barrier()
    draft_ms = [e[0].elapsed_time(e[1]) for e in evs]
    verify_ms = [e[1].elapsed_time(e[2]) for e in evs]
    commit_ms = [e[2].elapsed_time(e[3]) for e in evs]
    step_ms = [e[0].elapsed_time(e[3]) for e in evs]

    # correctness of what was timed: planted acceptance, no device-side errors
    if not (np.array_equal(accepted.cpu().numpy(), a_star) and int(flag.item()) == 0
            and das.workspace_status(ws) == 0):
        raise SystemExit("bench: device results failed their checks")

    K_bytes = K.numel() * K.element_size()
    draft_bytes = wl.prefix_bytes_per_layer() * L
    verify_bytes = wlv.prefix_bytes_per_layer() * L
    draft_s = sum(draft_ms) / 1e3
    draft_s, step_s = max_over_ranks([draft_s, sum(step_ms) / 1e3], world, dev)
    K_steps = args.steps
    gbs = whole_job_gbs(world, draft_bytes, K_steps, draft_s)
    tokens = int(wl.block_lens().sum())
    peak, peak_kind = peaks()
    per_launch_ms = statistics.mean(draft_ms) / L
    achieved = wl.prefix_bytes_per_layer() / (per_launch_ms / 1e3) / 1e9
    traffic = kernel_traffic(args.workload)

    e2e = None if args.no_e2e else e2e_arm(args, wl, cache, pl, P0, bl, ws, stream, dev)
    if e2e is not None and world > 1:
        (t,) = max_over_ranks([e2e.pop("_seconds")], world, dev)
        e2e["value"] = whole_job_gbs(world, draft_bytes, K_steps, t)
    elif e2e is not None:
        e2e.pop("_seconds")

    probes = seq = wave = f8 = commit = None
    if not args.no_probes:
        # the other workloads' attention phases, each on its full cache layout
        # (all R depth slabs allocated), and the long one again on a cache
        # compacted to the two slabs it reads (same bytes; layout effect)
        probes = {n: draft_probe(n, dev, 200, 5, peak, unflushed=(n == "decode"))
                  for n in ("long", "decode", "batched", "verify") if n != args.workload}
        probes["long_2slab"] = draft_probe("long", dev, 200, 5, peak, compact=True)
        commit = commit_probe("verify", dev, 200, 5, peak)
        # the single-sequence decode step's acceptance and commit ([1, 8, 32000])
        commit["decode"] = commit_probe("decode", dev, 200, 5, peak, vocab=32000)
        del cache, K, V
        torch.cuda.empty_cache()
        seq, wave = decode_cache_probes(dev, 20, 3, peak)
        f8 = {n: f8_probe(n, dev, 200, 5, peak) for n in ("decode", "long")}
        # against the bf16 cache on a layout like the e4m3 probe's (2 slabs for
        # long; the decode cache is small enough that its layout does not matter)
        for n, r in f8.items():
            ref = probes["long_2slab"] if n == "long" else probes.get(n)
            bf16_us = (ref["per_call_us"] if ref is not None
                       else statistics.mean(draft_ms) * 1e3 / L)
            r["speedup_vs_bf16_cache"] = round(bf16_us / r["per_call_us"], 3)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(wl, budget_s=12.0)

    line = {
        "metric": "Mature-V draft-attn prefix-KV GB/s (% of GB300 HBM peak); draft tokens/s",
        "value": round(gbs, 1),
        "unit": "GB/s",
        "n_gpus": world,
        "steps": K_steps,
        "warmup": args.warmup,
        "ms_per_step": round(statistics.mean(step_ms), 4),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (seeded depth-maturation law; no datasets or weights)",
        "config": {
            "workload": wl.name,
            "batch": B, "layers": L, "q_heads": wl.q_heads, "kv_heads": wl.kv_heads,
            "head_dim": wl.head_dim, "depths": R, "key_depth": wl.key_depth,
            "value_depth": wl.value_depth, "prefix_len": list(wl.prefix), "block": list(wl.block),
            "verify_width": W, "vocab": vocab, "seed": wl.seed,
            "parallelism": "replicas" if world > 1 else "single GPU",
            "cache_layout": f"all {R} depth slabs allocated "
                            f"({2 * K_bytes / 1e9:.1f} GB of K and V)",
            "l2": "flushed before every timed step (512 MiB written, then read back)",
        },
        "pct_of_hbm_peak": {(f"measured_copy_{peak:.1f}" if peak_kind == "measured"
                             else f"fallback_{peak:.0f}"):
                            round(100 * gbs / world / peak, 1),
                            "nominal_8000": round(100 * gbs / world / 8000.0, 1)},
        "draft_tokens_per_s": round(world * tokens * K_steps / draft_s, 1),
        "phases_ms": {"draft": round(statistics.mean(draft_ms), 4),
                      "verify": round(statistics.mean(verify_ms), 4),
                      "accept_append": round(statistics.mean(commit_ms), 4)},
        "verify_gbs": round(verify_bytes * K_steps / (sum(verify_ms) / 1e3) / 1e9, 1),
        "roofline": {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                     "frac": round(achieved / peak, 4), "traffic": traffic,
                     "kernel": "attn_kernel + merge_kernel (one Mature-V layer call)",
                     "peak_source": f"{peak_kind} HBM copy bandwidth"},
        "other_workloads": probes,
        "accept_append": commit,
        "sequential_draft": seq,
        "das_wave_refinement": wave,
        "e4m3_cache_draft": f8,
        "gpu_launches": K_steps * (launches_per_step or (2 * L * 2 + 2 + 2)),
        "gpu_launches_per_step": {"count": launches_per_step or (2 * L * 2 + 2 + 2),
                                  "source": "kernel nodes of the step's CUDA graphs"
                                  if launches_per_step else "launch sequence (two-kernel accept)"},
        "e2e": e2e,
        "cpu_baseline": cpu,
        "clocks": clocks.summary(),
        "wall_s": round(wall, 3),
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def draft_probe(name, dev, steps, warmup, peak, layers=0, compact=False, unflushed=False):
    """Per-call time of a workload's attention phase, timed like the main one
    (a CUDA graph of its L layer calls, L2 flushed before every replay), on
    the workload's full cache layout: all R depth slabs allocated, the read
    depths (kappa for keys, nu for values; depth R for both in a verify
    workload) holding the generator's values.  compact=True stores only the
    two slabs the calls read (the same bytes per call in a smaller cache).
    unflushed=True also times the graph replayed back to back without the
    flush, for a workload whose per-call bytes fit in L2 (decode: 67 MB per
    call against 129 MB of L2), reported beside the flushed figure."""
    import torch

    import paper_2609_34538_gb300 as das
    from synth import device as sdev
    from synth import workloads as wlm

    verify = wlm.WORKLOADS[name].kind == "verify"
    wl = wlm.WORKLOADS[name]
    if compact:
        wl = wl.replace(depths=2, key_depth=2 if verify else 1, value_depth=2)
    if layers:
        wl = wl.replace(layers=layers)
    L, B, W = wl.layers, wl.batch, wl.max_block
    stream = torch.cuda.Stream(device=dev)
    with torch.cuda.stream(stream):
        K, V = sdev.build_cache(wl, device=dev)
        cache = das.DepthKVCache(K, V)
        pl = torch.from_numpy(wl.prefix_lens()).to(dev)
        bl = torch.from_numpy(wl.block_lens()).to(dev)
        ws = das.new_workspace(cache, wl.q_heads, W, device=dev)
        ins = [sdev.layer_inputs(wl, l, dev) for l in range(L)]
        outs = [(torch.empty_like(q), torch.empty((B, wl.q_heads, W), dtype=torch.float32,
                                                  device=dev)) for q, _, _ in ins]
        flush = torch.empty(512 * 2 ** 20, dtype=torch.uint8, device=dev)
    stream.synchronize()

    def phase():
        for l, (q, kb, vb) in enumerate(ins):
            if verify:
                das.das_verify_attention(cache, l, wl.key_depth, pl, bl, q, kb, vb, ws,
                                         out=outs[l][0], lse=outs[l][1], stream=stream)
            else:
                das.das_mature_v_attention(cache, l, wl.key_depth, wl.value_depth, pl, bl, q, kb,
                                           vb, ws, out=outs[l][0], lse=outs[l][1], stream=stream)

    with torch.cuda.stream(stream):
        phase()
    stream.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        phase()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(warmup + steps)]
    for e0, e1 in ev:
        with torch.cuda.stream(stream):
            flush_l2(flush)
            e0.record(stream)
            g.replay()
            e1.record(stream)
    stream.synchronize()
    ms = [e0.elapsed_time(e1) for e0, e1 in ev[warmup:]]
    nbytes = wl.prefix_bytes_per_layer() * L
    gbs = nbytes * len(ms) / (sum(ms) / 1e3) / 1e9
    extra = {}
    if unflushed:
        ev2 = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(warmup + steps)]
        for e0, e1 in ev2:
            with torch.cuda.stream(stream):
                e0.record(stream)
                g.replay()
                e1.record(stream)
        stream.synchronize()
        ms2 = [e0.elapsed_time(e1) for e0, e1 in ev2[warmup:]]
        gbs2 = nbytes * len(ms2) / (sum(ms2) / 1e3) / 1e9
        extra = {"unflushed": {"per_call_us": round(statistics.mean(ms2) * 1e3 / L, 2),
                               "gbs": round(gbs2, 1), "pct_of_measured_hbm": round(100 * gbs2 / peak, 1),
                               "note": "graph replays back to back, L2 not flushed: part of "
                                       "each call's bytes may come from L2"}}
    if das.workspace_status(ws) != 0:
        raise SystemExit(f"bench: {name} attention phase reported a device-side error")
    cache_gb = 2 * K.numel() * K.element_size() / 1e9
    del K, V, cache, flush
    torch.cuda.empty_cache()
    return {"workload": wl.name,
            "cache_layout": (f"2 depth slabs ({cache_gb:.1f} GB of K and V)" if compact else
                             f"all {wl.depths} depth slabs ({cache_gb:.1f} GB of K and V)"),
            "bytes_per_call": wl.prefix_bytes_per_layer(),
            "per_call_us": round(statistics.mean(ms) * 1e3 / L, 2), "gbs": round(gbs, 1),
            "pct_of_measured_hbm": round(100 * gbs / peak, 1),
            "pct_of_nominal_8000": round(100 * gbs / 8000.0, 1),
            "draft_tokens_per_s": (None if verify else
                                   round(int(wl.block_lens().sum()) * len(ms) / (sum(ms) / 1e3), 1)),
            "steps": len(ms), **extra}


def commit_probe(name, dev, steps, warmup, peak, layers=0, calls=4, vocab=0):
    """Greedy acceptance and the commit at a verify-and-commit workload's
    shape (Sec. 3.4, App. B.1), each timed on its own as a CUDA graph of
    `calls` back-to-back calls on distinct inputs (L2 flushed before every
    replay; per-call time = graph time / calls): accept over fp32 logits
    [B][w][vocab] with planted acceptance lengths, then the append of
    n_b = min(a_b + 1, w) staged inputs' K/V at all R depths and L layers
    into the full cache (each call appends after the previous one).
    Algorithmic bytes per call: accept B * w * vocab * 4 (the logits read);
    append 2 (K and V) * sum_b n_b * R * L * Hkv * D * 2, read once and
    written once."""
    import torch

    import paper_2609_34538_gb300 as das
    from synth import device as sdev
    from synth import workloads as wlm

    wl = wlm.WORKLOADS[name]
    if layers:
        wl = wl.replace(layers=layers)
    if vocab or not wl.vocab:  # a draft workload's commit: logits of its block's rows
        wl = wl.replace(vocab=vocab or 32000)
    W, B = wl.max_block, wl.batch
    wl = wl.replace(extra_capacity=(calls - 1) * W)
    stream = torch.cuda.Stream(device=dev)
    with torch.cuda.stream(stream):
        K, V = sdev.build_cache(wl, key_depths=[], value_depths=[], device=dev)
        cache = das.DepthKVCache(K, V)
        staged = [sdev.build_staged(wl.replace(seed=wl.seed + c), W, device=dev)
                  for c in range(calls)]
        a_star, draft, logits = sdev.accept_tensors(wl, dev)
        logit_bufs = [logits] + [logits.clone() for _ in range(calls - 1)]
        P0 = torch.from_numpy(wl.prefix_lens()).to(dev)
        pl = P0.clone()
        acc = torch.empty(B, dtype=torch.int32, device=dev)
        tid = torch.empty((B, W), dtype=torch.int32, device=dev)
        nxt = torch.empty(B, dtype=torch.int32, device=dev)
        flag = torch.zeros(1, dtype=torch.int32, device=dev)
        flush = torch.empty(512 * 2 ** 20, dtype=torch.uint8, device=dev)
    stream.synchronize()

    def accept():
        for lg in logit_bufs:
            das.das_greedy_accept(lg, draft, acc, tid, nxt, stream=stream)

    def append():
        for kn, vn in staged:
            das.das_kv_append(cache, kn, vn, acc, pl, flag, stream=stream)

    with torch.cuda.stream(stream):
        accept()
        append()
        pl.copy_(P0)
    stream.synchronize()
    graphs = []
    for fn in (accept, append):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            fn()
        graphs.append(g)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)]
          for _ in range(warmup + steps)]
    for e in ev:
        with torch.cuda.stream(stream):
            pl.copy_(P0)
            flush_l2(flush)
            e[0].record(stream)
            graphs[0].replay()
            e[1].record(stream)
            graphs[1].replay()
            e[2].record(stream)
    stream.synchronize()
    n = np.minimum(a_star.astype(np.int64) + 1, W)
    if not (np.array_equal(acc.cpu().numpy(), a_star) and int(flag.item()) == 0
            and np.array_equal(pl.cpu().numpy(), wl.prefix_lens() + calls * n)):
        raise SystemExit("bench: accept / append results failed their checks")
    acc_ms = [e[0].elapsed_time(e[1]) / calls for e in ev[warmup:]]
    app_ms = [e[1].elapsed_time(e[2]) / calls for e in ev[warmup:]]
    acc_bytes = B * W * logits.shape[2] * 4
    app_bytes = 2 * int(n.sum()) * wl.depths * wl.layers * wl.kv_heads * wl.head_dim * 2 * 2
    del K, V, cache, staged, logit_bufs, flush
    torch.cuda.empty_cache()

    def rate(nbytes, ms):
        t = statistics.mean(ms)
        gbs = nbytes / (t / 1e3) / 1e9
        return {"us_per_call": round(t * 1e3, 2), "bytes_per_call": nbytes, "gbs": round(gbs, 1),
                "roofline": {"bound": "hbm", "achieved": round(gbs, 1), "peak": peak,
                             "unit": "GB/s", "frac": round(gbs / peak, 4)}}

    return {"workload": wl.name, "calls_per_graph": calls,
            "accept": {"shape": [B, W, int(logits.shape[2])], **rate(acc_bytes, acc_ms)},
            "append": {"positions_committed_per_call": int(n.sum()), "depths": wl.depths,
                       "layers": wl.layers, **rate(app_bytes, app_ms)},
            "steps": len(acc_ms)}


def decode_cache_probes(dev, steps, warmup, peak):
    """The sequential drafting loop and the DAS-Wave refinement on the
    single-sequence decode workload's full cache (all R depth slabs; keys
    exact at depths 1..r and R, values at R)."""
    import torch

    import paper_2609_34538_gb300 as das
    from synth import device as sdev
    from synth import workloads as wlm

    wl = wlm.WORKLOADS["decode"]
    stream = torch.cuda.Stream(device=dev)
    with torch.cuda.stream(stream):
        K, V = sdev.build_cache(wl, key_depths=set(range(1, wl.key_depth + 1)) | {wl.depths},
                                value_depths={wl.depths}, device=dev)
        cache = das.DepthKVCache(K, V)
        pl = torch.from_numpy(wl.prefix_lens()).to(dev)
        ws = das.new_workspace(cache, wl.q_heads, wl.max_block, device=dev)
    stream.synchronize()
    seq = sequential_probe(wl, cache, pl, ws, dev, steps, warmup, peak)
    wave = wave_probe(wl, cache, pl, dev, steps, warmup, peak)
    del K, V, cache
    torch.cuda.empty_cache()
    return seq, wave


def f8_probe(name, dev, steps, warmup, peak, layers=0):
    """Mature-V draft phase of workload `name` on the e4m3 cache variant
    (keys at depth r stored as e4m3, values at depth R as bf16; not in the
    paper), timed like the bf16 probes; bytes per call count 1 byte per key
    element and 2 per value element."""
    import torch

    import paper_2609_34538_gb300 as das
    from synth import device as sdev
    from synth import workloads as wlm

    wl = wlm.WORKLOADS[name].replace(depths=2, key_depth=1, value_depth=2)
    if layers:
        wl = wl.replace(layers=layers)
    L, B, W = wl.layers, wl.batch, wl.max_block
    stream = torch.cuda.Stream(device=dev)
    with torch.cuda.stream(stream):
        cache = das.DepthKVCacheF8.empty(2, L, B, wl.capacity, wl.kv_heads, wl.head_dim,
                                         device=dev)
        sdev.fill_matured(cache.v_top, wl.seed, 2, 1, 2, 2)
        sdev.fill_matured(cache.k_top, wl.seed, 1, 0, 2, 2)
        g = torch.Generator(device=dev).manual_seed(wl.seed)
        for t in (cache.k_low, cache.v_low):  # codes with exponent fields 4..9, random sign
            t.copy_(torch.randint(0x20, 0x50, t.shape, generator=g, device=dev, dtype=torch.int32)
                    .bitwise_or_(torch.randint(0, 2, t.shape, generator=g, device=dev,
                                               dtype=torch.int32) * 0x80).to(torch.uint8))
        pl = torch.from_numpy(wl.prefix_lens()).to(dev)
        bl = torch.from_numpy(wl.block_lens()).to(dev)
        ws = das.new_workspace_f8(cache, wl.q_heads, W, device=dev)
        ins = [sdev.layer_inputs(wl, l, dev) for l in range(L)]
        outs = [(torch.empty_like(q), torch.empty((B, wl.q_heads, W), dtype=torch.float32,
                                                  device=dev)) for q, _, _ in ins]
        flush = torch.empty(512 * 2 ** 20, dtype=torch.uint8, device=dev)
    stream.synchronize()

    def phase():
        for l, (q, kb, vb) in enumerate(ins):
            das.das_mature_v_attention_f8(cache, l, 1, 2, pl, bl, q, kb, vb, ws, out=outs[l][0],
                                          lse=outs[l][1], stream=stream)

    with torch.cuda.stream(stream):
        phase()
    stream.synchronize()
    gr = torch.cuda.CUDAGraph()
    with torch.cuda.graph(gr, stream=stream):
        phase()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(warmup + steps)]
    for e0, e1 in ev:
        with torch.cuda.stream(stream):
            flush_l2(flush)
            e0.record(stream)
            gr.replay()
            e1.record(stream)
    stream.synchronize()
    if das.workspace_status(ws) != 0:
        raise SystemExit(f"bench: e4m3 {name} probe reported a device-side error")
    ms = [e0.elapsed_time(e1) for e0, e1 in ev[warmup:]]
    nbytes = wl.prefix_bytes_per_layer() * 3 // 4 * L  # K 1 byte + V 2 bytes per element pair
    gbs = nbytes * len(ms) / (sum(ms) / 1e3) / 1e9
    del cache, flush
    torch.cuda.empty_cache()
    return {"workload": wl.name, "storage": "keys e4m3 (depth r), values bf16 (depth R)",
            "per_call_us": round(statistics.mean(ms) * 1e3 / L, 2), "gbs": round(gbs, 1),
            "pct_of_measured_hbm": round(100 * gbs / peak, 1), "steps": len(ms)}


def sequential_probe(wl, cache, pl, ws, dev, steps, warmup, peak):
    """The sequential drafting loop (Sec. 3.2, Eq. 4; App. A.2) on the main
    workload's cache: a block of T = max_block tokens drafted one at a time;
    token i runs d = key_depth recurrence steps x L layer calls with block
    length i, prefix values at depth R and prefix keys at depth s for step s
    (Mature-V) or at depth R (Deep K/V, Mature-Spec).  The T*d*L calls of one
    block are one CUDA graph; L2 is flushed before every replay."""
    import torch

    import paper_2609_34538_gb300 as das
    from synth import device as sdev

    L, B, T, R, d = wl.layers, wl.batch, wl.max_block, wl.depths, wl.key_depth
    stream = torch.cuda.Stream(device=dev)
    with torch.cuda.stream(stream):
        ins = [sdev.layer_inputs(wl, l, dev) for l in range(L)]
        outs = [(torch.empty_like(q), torch.empty((B, wl.q_heads, T), dtype=torch.float32,
                                                  device=dev)) for q, _, _ in ins]
        bls = [torch.full((B,), i, dtype=torch.int32, device=dev) for i in range(1, T + 1)]
        flush = torch.empty(512 * 2 ** 20, dtype=torch.uint8, device=dev)
    stream.synchronize()
    res = {}
    for policy in ("mature_v", "deep_kv"):
        calls = []
        for i in range(T):
            for s in range(1, d + 1):
                for l in range(L):
                    q, kb, vb = ins[l]
                    calls.append(das.AttentionCall(cache, pl, bls[i], q, kb, vb, ws,
                                                   out=outs[l][0], lse=outs[l][1]))
        kap = [s for i in range(T) for s in range(1, d + 1) for l in range(L)]

        def block():
            for c, k, l in zip(calls, kap, [l for _ in range(T * d) for l in range(L)]):
                c.mature_v(l, k if policy == "mature_v" else R, R, stream=stream)

        with torch.cuda.stream(stream):
            block()
        stream.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            block()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(warmup + steps)]
        for e0, e1 in ev:
            with torch.cuda.stream(stream):
                flush_l2(flush)
                e0.record(stream)
                g.replay()
                e1.record(stream)
        stream.synchronize()
        ms = [e0.elapsed_time(e1) for e0, e1 in ev[warmup:]]
        ncalls = T * d * L
        nbytes = wl.prefix_bytes_per_layer() * ncalls
        gbs = nbytes * len(ms) / (sum(ms) / 1e3) / 1e9
        res[policy] = {"us_per_token": round(statistics.mean(ms) * 1e3 / T, 1),
                       "us_per_call": round(statistics.mean(ms) * 1e3 / ncalls, 2),
                       "gbs": round(gbs, 1), "pct_of_measured_hbm": round(100 * gbs / peak, 1)}
    if das.workspace_status(ws) != 0:
        raise SystemExit("bench: sequential probe reported a device-side error")
    del flush
    return {"calls_per_block": T * d * L, "block_tokens": T, "recurrence_steps": d,
            "layers": L, **res}


def wave_probe(wl, cache, pl, dev, steps, warmup, peak, gamma=32, w_init=2, rounds=24, k=2,
               vocab=32000):
    """DAS-Wave carried parallel refinement (Sec. 3.3) on the main workload's
    cache with the paper's schedule (gamma 32, W_init 2, J 24; App. A.2) and
    k recurrent updates per round: J*k*L attention calls with Deep K/V prefix
    reads over W_j = min(gamma, W_init + j) active rows (Eq. 5), and J shifted
    readouts over [B][W_j][vocab] logits (Eq. 6).  Synthetic queries, block
    K/V and logits stand in for the looped model; one CUDA graph per
    refinement, L2 flushed before every replay."""
    import torch

    import paper_2609_34538_gb300 as das
    from synth import device as sdev

    L, B = wl.layers, wl.batch
    wg = wl.replace(block=(gamma,))
    stream = torch.cuda.Stream(device=dev)
    with torch.cuda.stream(stream):
        ins = [sdev.layer_inputs(wg, l, dev) for l in range(L)]
        outs = [(torch.empty_like(q), torch.empty((B, wl.q_heads, gamma), dtype=torch.float32,
                                                  device=dev)) for q, _, _ in ins]
        lbuf = [torch.randn((B, w, vocab), generator=torch.Generator(device=dev).manual_seed(w),
                            device=dev, dtype=torch.float32) * 2
                for w in range(1, gamma + 1)]
        ws = das.new_workspace(cache, wl.q_heads, gamma, device=dev)
        anchor = torch.zeros(B, dtype=torch.int32, device=dev)
        flush = torch.empty(512 * 2 ** 20, dtype=torch.uint8, device=dev)
    stream.synchronize()
    drv = das.WaveRefinement(cache, pl, ws, wl.q_heads, gamma=gamma, w_init=w_init,
                             rounds=rounds, k_steps=k)

    def step(j, s, layer):
        q, kb, vb = ins[layer]
        return q, kb, vb, outs[layer][0], outs[layer][1]

    def refine():
        drv.run(anchor, step, lambda j: lbuf[drv.widths[j] - 1], stream=stream)

    with torch.cuda.stream(stream):
        refine()
    stream.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        refine()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(warmup + steps)]
    for e0, e1 in ev:
        with torch.cuda.stream(stream):
            flush_l2(flush)
            e0.record(stream)
            g.replay()
            e1.record(stream)
    stream.synchronize()
    if das.workspace_status(ws) != 0:
        raise SystemExit("bench: DAS-Wave probe reported a device-side error")
    ms = [e0.elapsed_time(e1) for e0, e1 in ev[warmup:]]
    ncalls = rounds * k * L
    nbytes = wl.replace(key_depth=wl.depths).prefix_bytes_per_layer() * ncalls
    gbs = nbytes * len(ms) / (sum(ms) / 1e3) / 1e9
    del flush, lbuf
    return {"gamma": gamma, "w_init": w_init, "rounds": rounds, "k": k,
            "attention_calls": ncalls, "readouts": rounds,
            "widths": [drv.widths[0], drv.widths[-1]],
            "us_per_refinement": round(statistics.mean(ms) * 1e3, 1),
            "us_per_call": round(statistics.mean(ms) * 1e3 / (ncalls + rounds), 2),
            "attention_gbs": round(gbs, 1), "pct_of_measured_hbm": round(100 * gbs / peak, 1)}


def e2e_arm(args, wl, cache, pl, P0, bl, ws, stream, dev):
    """The draft phase through the public API with host buffers, pipelined as
    a serving loop would run it.  Every step copies the step's queries and
    block K/V of all L layers from one pinned host buffer to the device (one
    copy), runs the L layer calls (AttentionCall objects built once) and
    copies all outputs and lse back to pinned host memory (one copy).  The
    copies run on a second stream into double-buffered device memory, so the
    copies of steps s-1 and s+1 overlap the calls of step s; the timed region
    runs from before the first input copy to the end of the last output copy."""
    import torch

    import paper_2609_34538_gb300 as das
    from synth import workloads as wlm

    L, B, W = wl.layers, wl.batch, wl.max_block
    al = lambda n: (n + 255) // 256 * 256
    q_shape, kv_shape = (B, W, wl.q_heads, wl.head_dim), (B, W, wl.kv_heads, wl.head_dim)
    lse_shape = (B, wl.q_heads, W)
    nq, nkv = al(int(np.prod(q_shape)) * 2), al(int(np.prod(kv_shape)) * 2)
    nlse = al(int(np.prod(lse_shape)) * 4)
    in_per, out_per = nq + 2 * nkv, nq + nlse
    host_in = torch.empty(L * in_per, dtype=torch.uint8).pin_memory()
    host_out = [torch.empty(L * out_per, dtype=torch.uint8).pin_memory() for _ in range(2)]
    dev_in = [torch.empty(L * in_per, dtype=torch.uint8, device=dev) for _ in range(2)]
    dev_out = [torch.empty(L * out_per, dtype=torch.uint8, device=dev) for _ in range(2)]

    def view(buf, off, dtype, shape):
        n = int(np.prod(shape)) * torch.tensor([], dtype=dtype).element_size()
        return buf[off:off + n].view(dtype).view(shape)

    for l in range(L):
        base = l * in_per
        q = wlm.gen_q(wl, l)
        kb, vb = wlm.gen_block_kv(wl, l)
        for off, x, shp in ((base, q, q_shape), (base + nq, kb, kv_shape),
                            (base + nq + nkv, vb, kv_shape)):
            view(host_in, off, torch.int16, shp).copy_(torch.from_numpy(x.view(np.int16)))
    calls = [[], []]
    for k in range(2):
        for l in range(L):
            base, ob = l * in_per, l * out_per
            calls[k].append(das.AttentionCall(
                cache, pl, bl, view(dev_in[k], base, torch.bfloat16, q_shape),
                view(dev_in[k], base + nq, torch.bfloat16, kv_shape),
                view(dev_in[k], base + nq + nkv, torch.bfloat16, kv_shape), ws,
                out=view(dev_out[k], ob, torch.bfloat16, q_shape),
                lse=view(dev_out[k], ob + nq, torch.float32, lse_shape)))
    bi, bo = host_in.numel(), host_out[0].numel()
    cs = torch.cuda.Stream(device=dev)

    def run(n):
        """n steps; returns (start event on cs, end event on cs)."""
        ev_in = [torch.cuda.Event() for _ in range(n)]
        ev_done = [torch.cuda.Event() for _ in range(n)]
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        cs.wait_stream(stream)
        e0.record(cs)
        for s in range(min(2, n)):  # inputs of the first two steps
            with torch.cuda.stream(cs):
                dev_in[s % 2].copy_(host_in, non_blocking=True)
            ev_in[s].record(cs)
        for s in range(n):
            k = s % 2
            stream.wait_event(ev_in[s])
            for l, c in enumerate(calls[k]):
                c.mature_v(l, wl.key_depth, wl.value_depth, stream=stream)
            ev_done[s].record(stream)
            cs.wait_event(ev_done[s])
            with torch.cuda.stream(cs):
                host_out[k].copy_(dev_out[k], non_blocking=True)  # outputs of step s
                if s + 2 < n:                                    # inputs of step s + 2
                    dev_in[k].copy_(host_in, non_blocking=True)
            if s + 2 < n:
                ev_in[s + 2].record(cs)
        e1.record(cs)
        return e0, e1

    with torch.cuda.stream(stream):
        pl.copy_(P0)
    run(max(args.warmup, 2))
    torch.cuda.synchronize(dev)
    e0, e1 = run(args.steps)
    e1.synchronize()
    secs = e0.elapsed_time(e1) / 1e3
    draft_bytes = wl.prefix_bytes_per_layer() * L
    return {"value": round(draft_bytes * args.steps / secs / 1e9, 1), "unit": "GB/s",
            "h2d_bytes_per_step": bi, "d2h_bytes_per_step": bo,
            "note": "per step one pinned H2D copy of all layers' inputs and one D2H copy of "
                    "all outputs, on a copy stream overlapping the neighbouring steps' calls; "
                    f"L2 not flushed between e2e steps: a step streams {draft_bytes / 1e9:.2f} GB "
                    "of cache, " + (f"{draft_bytes / 129e6:.0f}x the 129 MB L2"
                                   if draft_bytes > 129e6 else "which fits in the 129 MB L2"),
            "_seconds": secs}


# ----------------------------------------------------------------------------- CPU legs

def oracle_sample(wl, heads):
    """Host inputs of the draft phase restricted to the first `heads` kv heads:
    a 2-slab cache (slab 1 = keys at depth r, slab 2 = values at depth R)."""
    from synth import T_KCACHE, T_VCACHE, matured_block
    from synth import workloads as wlm
    sub = wl.replace(kv_heads=heads, q_heads=heads * wl.group)
    P = sub.prefix_lens()
    shape = (2, sub.layers, sub.batch, int(P.max()) if P.max() > 0 else 1, heads, sub.head_dim)
    K = np.zeros(shape, dtype=np.uint16)
    V = np.zeros(shape, dtype=np.uint16)
    for l in range(sub.layers):
        for b in range(sub.batch):
            n = int(P[b])
            K[0, l, b, :n] = matured_block(sub.seed, T_KCACHE, 0, sub.key_depth, sub.depths, l, b,
                                           0, n, 0, heads, sub.head_dim)
            V[1, l, b, :n] = matured_block(sub.seed, T_VCACHE, 1, sub.value_depth, sub.depths, l,
                                           b, 0, n, 0, heads, sub.head_dim)
    ins = []
    for l in range(sub.layers):
        kb, vb = wlm.gen_block_kv(sub, l)
        ins.append((wlm.gen_q(sub, l), kb, vb))
    return sub, K, V, P, sub.block_lens(), ins


def time_oracle(sub, K, V, P, T, ins, budget_s, min_reps=1):
    import oracle
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    reps, t0 = 0, time.perf_counter()
    while reps < min_reps or time.perf_counter() - t0 < budget_s:
        for l, (q, kb, vb) in enumerate(ins):
            oracle.attention(K, V, l, 1, 2, P, T, q, kb, vb, nthreads=cores)
        reps += 1
    secs = time.perf_counter() - t0
    nbytes = int(P.astype(np.int64).sum()) * sub.kv_heads * sub.head_dim * 4 * sub.layers * reps
    return nbytes / secs / 1e9, secs, reps, cores


def sample_heads(wl, target_s=12.0):
    """kv heads of the draft phase that the oracle covers in about target_s."""
    return max(1, min(wl.kv_heads, 4 if wl.max_prefix > 10000 else wl.kv_heads))


def cpu_baseline(wl, budget_s=12.0):
    heads = sample_heads(wl)
    sub, K, V, P, T, ins = oracle_sample(wl, heads)
    gbs, secs, reps, cores = time_oracle(sub, K, V, P, T, ins, budget_s)
    return {"value": round(gbs, 4), "unit": "GB/s", "cores": cores, "kind": "oracle",
            "sample": f"draft phase (all {wl.layers} layers) restricted to kv heads 0..{heads - 1} "
                      f"of {wl.kv_heads}, repeated {reps}x in {secs:.1f} s; fp64, threaded over "
                      "(sequence, query head)"}


def reference_arm(args):
    """The fp64 oracle on the host cores, on the same workload, metric and unit.
    Each step is a bounded sample (one layer call over the first kv heads),
    sized so that warmup + steps take about a minute in all."""
    rank, world, _ = dist_env()
    if rank != 0:
        return
    from synth import workloads as wlm
    wl = wlm.WORKLOADS[args.workload]
    if args.layers:
        wl = wl.replace(layers=args.layers)
    budget = 60.0 / max(1, args.steps + args.warmup)
    # time one kv head of one layer, then scale the sample to the budget
    probe = wl.replace(layers=1)
    sub, K, V, P, T, ins = oracle_sample(probe, 1)
    _, t1, _, cores = time_oracle(sub, K, V, P, T, ins[:1], 0.0)
    heads = int(max(1, min(wl.kv_heads, budget / max(t1, 1e-6))))
    sub, K, V, P, T, ins = oracle_sample(probe, heads)
    for _ in range(args.warmup):
        time_oracle(sub, K, V, P, T, ins[:1], 0.0)
    per_step = []
    for _ in range(args.steps):
        _, secs, _, cores = time_oracle(sub, K, V, P, T, ins[:1], 0.0)
        per_step.append(secs)
    nbytes = int(P.astype(np.int64).sum()) * heads * wl.head_dim * 4
    value = nbytes * args.steps / sum(per_step) / 1e9
    sample = (f"per step: one Mature-V layer call restricted to kv heads 0..{heads - 1} of "
              f"{wl.kv_heads}; fp64 oracle threaded over (sequence, query head)")
    line = {"impl": "reference", "metric": "Mature-V draft-attn prefix-KV GB/s (% of GB300 HBM "
            "peak); draft tokens/s", "value": round(value, 4), "unit": "GB/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(1e3 * statistics.mean(per_step), 3), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": wl.name, "sample_kv_heads": heads},
            "cpu_baseline": {"value": round(value, 4), "unit": "GB/s", "cores": cores,
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": round(value, 4), "unit": "GB/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    args = parse()
    if args.impl == "reference":
        reference_arm(args)
    else:
        gpu_arm(args)


if __name__ == "__main__":
    main()
