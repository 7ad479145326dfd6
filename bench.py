#!/usr/bin/env python
"""Pruned ViT forward throughput on GB300 through the libdora C ABI.

Workload (default): DeiT-Base shape, batch 256 per GPU, 197 tokens, D=768,
12 heads, MLP 3072, 12 blocks, hard pruning at blocks 3/6/9 with per-image
removal counts drawn so the batch-mean token-layer compression (Eq. 4) is
about 0.38; deletion scores are synthetic per-image tables keyed by original
token id.  One step = one forward of the whole batch: at each pruning block
the score gather (actor stand-in) and dora_pruned_block, elsewhere
dora_pruned_block without deletion.

``--config cfg6`` runs the DINOv2-B/14 shape instead (257 tokens, LayerScale
folded into the attention-output and fc2 weights at load, 14-pixel patches
and the LC1 head in the complete-forward leg).

Prints one JSON line.  ``--impl reference`` times the fp64 CPU oracle on the
same workload instead (bounded samples, host cores only).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import dora_synth as S  # noqa: E402
from paper_2609_34325_gb300 import accounting as A  # noqa: E402

METRIC = "pruned ViT forward images/sec on 1 GB300; varlen-attn % bf16 peak; compact GB/s"
UNIT = "images/s"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}

# buffer sets the end-to-end leg rotates (inputs uploaded, outputs read back)
E2E_SETS = 3

# DRAM traffic of the GEMM (dram__bytes_read.sum + dram__bytes_write.sum)
# from an ncu capture of the linear micro-benchmark (50432 rows, D = 768, MLP
# 3072: one launch of each linear, inputs far above L2), keyed by the sha256 of
# the kernel source it was taken on: bytes per row of each linear.  The bench
# scales it to its own launches by their row counts (weights are read once a
# launch, a small share), so it is reported for the DeiT-B shape only, and as
# null once the source changes.
NCU_GEMM_BYTES_PER_ROW = {
    # profiles/gemm_tcgen05_deit_base_b256.md
    "3834b88b7bfb10b6fa882df991368856ad442bb685159ae83f4cbf3d74e9e6e0": {
        "gemm_qkv": 5140.8, "gemm_proj": 4038.6, "gemm_fc1": 6636.2, "gemm_fc2": 9222.7},
}


# DRAM traffic of one launch of the fused selection + compaction, from an ncu
# capture (dram__bytes_read.sum + dram__bytes_write.sum) of the token
# micro-benchmark's DeiT-B case (inputs cycled beyond 2 x L2), keyed by the
# sha256 of the kernel source; null once the source changes.
NCU_TRAFFIC_SELECT_COMPACT = {
    # profiles/select_compact_tokens.md: mean of 3 launches, 256 x 197 tokens,
    # D = 768, 34,284 rows kept (106.5 MB algorithmic)
    # (re-keyed after a comment-only edit; the compiled kernel is bit-identical)
    "574dbcc5d5ca29fa8d44aca95296f78a0ac7923926d3d4a15804b7494abe9505": {
        "traffic": 59518976, "case": "micro-benchmark: 256 x 197 tokens, D = 768, 34284 kept "
                                     "rows, inputs cycled beyond 2 x L2"},
}


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", default="cfg3")
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--input-sets", type=int, default=3)
    ap.add_argument("--cpu-images", type=int, default=20)
    ap.add_argument("--no-extras", action="store_true",
                    help="headline loop only (no dense, e2e, per-kernel or CPU legs)")
    ap.add_argument("--graph", action="store_true", help="replay the step as a CUDA graph")
    ap.add_argument("--split", type=int, default=1,
                    help="run the batch as this many independent sub-batches on as many streams")
    return ap.parse_args()


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return {k: float(d[k]) for k in FALLBACK_PEAKS}, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


def sha256_of(path):
    with open(path, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()


# ---------------------------------------------------------------------------
# workload (host side, shared by both arms)
# ---------------------------------------------------------------------------
class HostWorkload:
    """Seeded inputs of one workload.  With ``host_tensors`` False only the
    deletion schedule and score tables are made here (they fix the workload's
    structure); activations and weights are then drawn on the device with the
    same distributions (see device_tensors), which keeps the set-up of the
    large extra workloads to seconds."""

    def __init__(self, cfg, seed, n_sets, host_tensors=True):
        self.cfg = cfg
        self.seed = seed
        self.cu0, self.ids0 = S.initial_layout(cfg)
        self.sets = []
        for r in range(n_sets):
            s = seed + 7919 * r
            keeps, befores = S.keep_schedule(cfg, s)
            tables = [S.score_table(cfg, blk, s) for blk in cfg.prune_blocks]
            self.sets.append(dict(seed=s, x=S.activations_bf16(cfg, s) if host_tensors else None,
                                  keeps=keeps, befores=befores, tables=tables))
        self.weights = ([S.block_weights(cfg, l, seed) for l in range(cfg.depth)]
                        if host_tensors else None)

    def lengths_per_block(self, r):
        """Token count of every image entering each block, for set r."""
        cfg = self.cfg
        sched = dict(zip(cfg.prune_blocks, self.sets[r]["keeps"]))
        n = np.full(cfg.batch, cfg.n_tokens, dtype=np.int64)
        out = []
        for l in range(cfg.depth):
            m = sched[l].astype(np.int64) if l in sched else n
            out.append((n.copy(), m.copy()))
            n = m
        return out


# ---------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id):
        self.lines, self.proc, self.gpu_id = [], None, gpu_id

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", self.gpu_id, "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "20"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except OSError:
            self.proc = None

    def _read(self):
        for ln in self.proc.stdout:
            self.lines.append((time.time(), ln.strip()))

    def stop(self, t0, t1):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=2)
        return clock_summary(self.lines, t0, t1)


def clock_summary(lines, t0, t1):
    """Median SM clock, the maximum clock and the throttle reasons seen in the
    (arrival time, nvidia-smi CSV line) samples that fall in [t0, t1] (with a
    little slack for the sampler's latency); lines that do not parse are
    skipped."""
    sm, mx, reasons = [], None, set()
    for ts, ln in lines:
        f = [x.strip() for x in ln.split(",")]
        if len(f) < 9 or not (t0 - 0.05 <= ts <= t1 + 0.15):
            continue
        try:
            sm.append(float(f[1]))
            mx = float(f[2])
        except ValueError:
            continue
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for name, v in zip(names, f[5:9]):
            if v.lower().startswith("active"):
                reasons.add(name)
    if not sm:
        return {"sm_mhz": None, "sm_max_mhz": mx, "reasons": [], "samples": 0}
    return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
            "samples": len(sm)}


def device_tensors(torch, cfg, seed, n_sets, dev):
    """Block weights (nn.Linear layout, bf16 N(0, 0.02^2), biases 0, LayerNorm
    gamma 1, beta 0) and N(0, 1) activations of every input set, drawn on the
    device from a seeded torch generator: the distributions of dora_synth's
    host generator, without its host-side cost at ViT-L size."""
    g = torch.Generator(device=dev)
    g.manual_seed(int(seed))
    d, m = cfg.dim, cfg.mlp_dim
    bf16 = torch.bfloat16

    def normal(shape, std):
        return (torch.randn(shape, generator=g, device=dev, dtype=torch.float32) * std).to(bf16)

    blocks = []
    for _ in range(cfg.depth):
        blocks.append({
            "ln1_w": torch.ones(d, dtype=bf16, device=dev),
            "ln1_b": torch.zeros(d, dtype=bf16, device=dev),
            "w_qkv": normal((3 * d, d), 0.02), "b_qkv": torch.zeros(3 * d, dtype=bf16, device=dev),
            "w_proj": normal((d, d), 0.02), "b_proj": torch.zeros(d, dtype=bf16, device=dev),
            "ln2_w": torch.ones(d, dtype=bf16, device=dev),
            "ln2_b": torch.zeros(d, dtype=bf16, device=dev),
            "w_fc1": normal((m, d), 0.02), "b_fc1": torch.zeros(m, dtype=bf16, device=dev),
            "w_fc2": normal((d, m), 0.02), "b_fc2": torch.zeros(d, dtype=bf16, device=dev)})
        if cfg.layerscale:
            # per-channel LayerScale on both branches (folded into w_proj and
            # w_fc2 at load), gamma ~ 0.05 + 0.45 U(0, 1) as the host generator draws it
            for nm in ("ls1", "ls2"):
                u = torch.rand(d, generator=g, device=dev, dtype=torch.float32)
                blocks[-1][nm] = (0.05 + 0.45 * u).to(bf16)
    xs = [normal((cfg.batch * cfg.n_tokens, d), 1.0) for _ in range(n_sets)]
    return blocks, xs


def workload_config(cfg, world, nsets, graph=False, streams=1):
    """The bench line's ``config``: the same for both arms."""
    return {
        "workload": f"{cfg.name}: batch {cfg.batch}/GPU, N={cfg.n_tokens}, "
                    f"D={cfg.dim}, H={cfg.heads}, MLP {cfg.mlp_dim}, {cfg.depth} blocks, "
                    f"prune at {'/'.join(map(str, cfg.prune_blocks))}",
        "global_batch": cfg.batch * world, "seq_len": cfg.n_tokens,
        "parallelism": f"dp{world} (independent replicas, no collective)",
        "l2": f"{nsets} input sets cycled; each step also streams ~1 GB of weights and "
              "intermediates, far above the 129 MB L2",
        "cuda_graph": bool(graph),
        "streams": streams,
    }


def gpu_uuid_arg(torch, dev_index):
    try:
        u = str(torch.cuda.get_device_properties(dev_index).uuid)
        return u if u.startswith("GPU-") else "GPU-" + u
    except Exception:
        return str(dev_index)


# the other forward shapes timed beside the main workload (pruned, dense and
# the per-kernel pass): ViT-L/16, ViT-B/16 at 384 pixels and DINOv2-B/14
EXTRA_WORKLOADS = ("cfg4", "cfg5", "cfg6")


def run_gpu(args, rank, world, local_rank):
    import torch

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    stream = torch.cuda.Stream(device=dev)
    with torch.cuda.stream(stream):
        res, hw = _run_gpu_on_stream(args, rank, world, local_rank, dev, stream, args.config)
        if not args.no_extras and args.config == "cfg3" and args.split == 1 and not args.graph:
            res["workloads"] = {}
            for name in EXTRA_WORKLOADS:
                sub, _ = _run_gpu_on_stream(args, rank, world, local_rank, dev, stream, name,
                                            core=True)
                res["workloads"][name] = sub
                torch.cuda.empty_cache()
        return res, hw


def _run_gpu_on_stream(args, rank, world, local_rank, dev, stream, cfg_name, core=False):
    """The bench legs of one workload.  ``core``: the pruned and dense
    forwards and the per-kernel pass only, with device-drawn weights and
    activations (the extra workloads)."""
    import torch
    import paper_2609_34325_gb300 as P

    P.load_library()
    cfg = S.get_config(cfg_name)
    peaks, peak_src = load_peaks()
    nsets_arg = 2 if core else args.input_sets
    hw = HostWorkload(cfg, args.seed + 100003 * rank, nsets_arg, host_tensors=not core)
    t_cap = cfg.batch * cfg.n_tokens

    def bf(a):
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).to(dev)

    def i32(a):
        return torch.from_numpy(np.ascontiguousarray(a, dtype=np.int32)).to(dev)

    # weights as a deployment loads them: LayerNorm affines folded into the QKV
    # and fc1 weights once (dora_fold_block_weights), outside the step
    if core:
        wdev, xdev = device_tensors(torch, cfg, hw.seed, nsets_arg, dev)
    else:
        wdev = [{k: bf(v) for k, v in w.items()} for w in hw.weights]
        xdev = [bf(s_["x"]) for s_ in hw.sets]
    blocks = [P.BlockWeights(w, cfg.dim, cfg.heads, cfg.mlp_dim, cfg.ln_eps).fold(stream)
              for w in wdev]
    torch.cuda.synchronize()
    sets = [dict(x=xdev[r], keeps=[i32(k) for k in s["keeps"]],
                 tables=[torch.from_numpy(t).to(dev) for t in s["tables"]])
            for r, s in enumerate(hw.sets)]
    # The batch runs as `split` independent sub-batches of whole images, each
    # on its own stream with its own boundaries, ids, row moments and
    # workspace: the kernels are persistent over all SMs, so one lane's next
    # kernel starts on the SMs another lane's kernel frees in its last wave.
    split = max(1, min(args.split, cfg.batch))
    edges = [round(k * cfg.batch / split) for k in range(split + 1)]
    lanes = []
    for k in range(split):
        i0, i1 = edges[k], edges[k + 1]
        r0, r1 = int(hw.cu0[i0]), int(hw.cu0[i1])
        tc, nb = r1 - r0, i1 - i0
        L = dict(i0=i0, i1=i1, r0=r0, r1=r1, tcap=tc, nb=nb,
                 stream=stream if k == 0 else torch.cuda.Stream(device=dev),
                 cu0=i32(hw.cu0[i0:i1 + 1] - r0), ids0=i32(hw.ids0[r0:r1]),
                 ws=P.alloc_workspace(tc, nb, blocks[0], dev),
                 scores=torch.zeros(tc, dtype=torch.float32, device=dev),
                 kept=torch.zeros(tc, dtype=torch.int32, device=dev))
        # E2E_SETS sets of buffers: the e2e pipeline rotates them between steps
        # so that a step's readback never races a later step's writes
        L["xbufs"] = [[torch.zeros(tc, cfg.dim, dtype=torch.bfloat16, device=dev)
                       for _ in range(2)] for _ in range(E2E_SETS)]
        L["cubufs"] = [[torch.zeros(nb + 1, dtype=torch.int32, device=dev) for _ in range(2)]
                       for _ in range(E2E_SETS)]
        L["idbufs"] = [[torch.zeros(tc, dtype=torch.int32, device=dev) for _ in range(2)]
                       for _ in range(E2E_SETS)]
        # row moments handed from block to block (x_out_moments -> x_in_moments)
        L["mvbufs"] = [[torch.zeros(tc, 2, dtype=torch.float32, device=dev) for _ in range(2)]
                       for _ in range(E2E_SETS)]
        lanes.append(L)
    ws = lanes[0]["ws"]
    prune = list(cfg.prune_blocks)
    # the deployment actor at random init (Sec. 3.2), for the leg whose
    # deletion scores come from the actor (the configured keep counts stay)
    actor = None
    if not args.no_extras and not core:
        wa = S.actor_weights(cfg.dim, cfg.depth, cfg.n_vis0, args.seed)
        actor = P.ActorWeights({k: bf(v) for k, v in wa.items()}, cfg.dim, cfg.depth,
                               cfg.n_vis0).prepare(stream)
        for L in lanes:
            nb, tc = L["nb"], L["tcap"]
            L["actor"] = dict(
                ws=P.alloc_actor_workspace(tc, nb, actor, dev),
                rho=torch.zeros(nb, dtype=torch.float32, device=dev),
                e=torch.zeros(nb, dtype=torch.int32, device=dev),
                out=[torch.zeros(nb, dtype=torch.int32, device=dev) for _ in range(4)],
                scores=torch.zeros(tc, dtype=torch.float32, device=dev))
    launches_per_step = {True: 0, False: 0}

    def forward(inp, pruned=True, pair=0, with_actor=False):
        """One forward step: every lane through the 12 blocks, block launches
        interleaved across lanes; the main stream joins the others at the end.
        Returns [(x_out, cu_out)] per lane."""
        if split > 1:
            e = torch.cuda.Event()
            e.record(stream)
            for L in lanes[1:]:
                L["stream"].wait_event(e)
        st = []
        for L in lanes:
            st.append(dict(x=inp["x"][L["r0"]:L["r1"]], cu=L["cu0"], ids=L["ids0"], mv=None))
        n = 0
        for l in range(cfg.depth):
            for L, c in zip(lanes, st):
                xbuf, cubuf, idbuf, mvbuf = (L["xbufs"][pair], L["cubufs"][pair],
                                             L["idbufs"][pair], L["mvbufs"][pair])
                out = xbuf[l % 2]
                mv_out = mvbuf[l % 2] if l + 1 < cfg.depth else None
                # QKV, attention, projection, fc1, fc2, the merge of the
                # projection's moments (the compaction merges them for the kept
                # rows at a pruning block) (+ row moments of the first input, +
                # merge of the output's moments)
                n += 5 + (not (pruned and l in prune)) + (c["mv"] is None) + (mv_out is not None)
                sl = L["stream"]
                if pruned and l in prune and with_actor:
                    j = prune.index(l)
                    A_ = L["actor"]
                    P.dora_pruned_block_actor(c["x"], c["cu"], blocks[l], cfg.n_tokens, out,
                                              L["ws"], actor, l, A_["rho"], A_["e"], *A_["out"],
                                              A_["scores"], A_["ws"], c["ids"], cubuf[j % 2],
                                              idbuf[j % 2],
                                              keep_counts=inp["keeps"][j][L["i0"]:L["i1"]],
                                              kept_idx=L["kept"], x_in_moments=c["mv"],
                                              x_out_moments=mv_out, stream=sl)
                    c["cu"], c["ids"] = cubuf[j % 2], idbuf[j % 2]
                    # actor: input projection, gate, LayerNorm statistics, QKV,
                    # attention, output projection, moment merge, two
                    # feed-forward linears, the selector's first linear, budget
                    # and selector; then the selection fused with the compaction
                    n += 12 + 1
                elif pruned and l in prune:
                    j = prune.index(l)
                    P.dora_gather_scores(inp["tables"][j][L["i0"]:L["i1"]], c["ids"], c["cu"],
                                         L["scores"], stream=sl)
                    P.dora_pruned_block(c["x"], c["cu"], blocks[l], cfg.n_tokens, out, L["ws"],
                                        ids_in=c["ids"], scores=L["scores"],
                                        keep_counts=inp["keeps"][j][L["i0"]:L["i1"]],
                                        cu_out=cubuf[j % 2], ids_out=idbuf[j % 2],
                                        kept_idx=L["kept"], x_in_moments=c["mv"],
                                        x_out_moments=mv_out, stream=sl)
                    c["cu"], c["ids"] = cubuf[j % 2], idbuf[j % 2]
                    n += 2                         # gather, selection + compaction
                else:
                    P.dora_pruned_block(c["x"], c["cu"], blocks[l], cfg.n_tokens, out, L["ws"],
                                        ids_in=c["ids"], x_in_moments=c["mv"],
                                        x_out_moments=mv_out, stream=sl)
                c["x"], c["mv"] = out, mv_out
        for L in lanes[1:]:
            e = torch.cuda.Event()
            e.record(L["stream"])
            stream.wait_event(e)
        launches_per_step[pruned] = n
        return [(c["x"], c["cu"]) for c in st]

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()

    def max_over_ranks(v):
        if world == 1:
            return v
        import torch.distributed as dist
        t = torch.tensor([v], dtype=torch.float64, device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        return float(t.item())

    def timed(step_fn, steps, warmup, sample_clocks=False):
        for i in range(warmup):
            step_fn(i)
        torch.cuda.synchronize()
        sampler = ClockSampler(gpu_uuid_arg(torch, local_rank)) if sample_clocks else None
        if sampler:
            sampler.start()
            time.sleep(0.4)
        barrier()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        w0 = time.time()
        e0.record(stream)
        for i in range(steps):
            step_fn(i)
        e1.record(stream)
        torch.cuda.synchronize()
        w1 = time.time()
        barrier()
        ms = e0.elapsed_time(e1)
        clocks = sampler.stop(w0, w1) if sampler else None
        return max_over_ranks(ms / 1000.0), clocks

    nsets = len(sets)
    graph = None
    if args.graph:
        # one graph per input set: the step is launch-only and capture-safe
        graphs = []
        for r in range(nsets):
            forward(sets[r])
            torch.cuda.synchronize()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                forward(sets[r])
            graphs.append(g)
        graph = graphs

    def step_pruned(i):
        if graph is not None:
            graph[i % nsets].replay()
        else:
            forward(sets[i % nsets], True)

    secs, clocks = timed(step_pruned, args.steps, max(args.warmup, 3), sample_clocks=True)
    images = cfg.batch * args.steps * world
    value = images / secs
    st = max(P.dora_read_status(P.dora_workspace_status(L["ws"])) for L in lanes)
    result = {
        "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": max(args.warmup, 3),
        "ms_per_step": round(1000 * secs / args.steps, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded bf16 N(0,1) activations, N(0,0.02) weights, U(0,1) score "
                "tables); no trained weights or images",
        "config": workload_config(cfg, world, nsets, args.graph, split),
        "clocks": clocks,
        "gpu_launches": launches_per_step[True] * args.steps,
        "device_status": st,
    }
    if args.no_extras:
        return result, None

    # unpruned dense forward: same kernels, no deletion
    dsecs, _ = timed(lambda i: forward(sets[i % nsets], False), args.steps,
                     max(args.warmup, 3))
    result["dense"] = {"value": round(cfg.batch * args.steps * world / dsecs, 1), "unit": UNIT,
                       "ms_per_step": round(1000 * dsecs / args.steps, 4)}
    result["speedup_vs_dense"] = round(dsecs / secs, 4)
    if core:
        # the extra workloads: the per-kernel pass for the rooflines, then done
        kern = profile_kernels(torch, P, cfg, hw, sets, blocks, dev, stream, t_cap,
                               steps=max(3, min(args.steps, 20)))
        rep = roofline_report(kern, peaks, peak_src, cfg_name)
        keeps = hw.sets[0]["keeps"]
        sched = dict(zip(cfg.prune_blocks, keeps))
        fl = A.trajectory_flops(cfg.depth, cfg.dim, cfg.mlp_dim, cfg.n_tokens, sched)
        fd = A.trajectory_flops(cfg.depth, cfg.dim, cfg.mlp_dim, cfg.n_tokens, {})
        out = {k: result[k] for k in ("value", "unit", "ms_per_step", "config", "clocks",
                                      "gpu_launches", "device_status", "dense",
                                      "speedup_vs_dense")}
        out["data"] = ("synthetic: deletion schedule and score tables from the seeded host "
                       "generator; bf16 N(0,1) activations and N(0,0.02) weights drawn on the "
                       "device by a seeded torch generator")
        out.update({k: rep[k] for k in ("roofline", "roofline_attention", "roofline_compact",
                                        "kernels")})
        out["workload_stats"] = {
            "compression_C_mean": round(float(S.compression_from_counts(
                cfg, keeps, hw.sets[0]["befores"]).mean()), 4),
            "block_gflops_per_image_pruned": round(float(fl.mean()) / 1e9, 3),
            "block_gflops_per_image_dense": round(float(fd.mean()) / 1e9, 3)}
        return out, hw

    # the same pruned forward with the actor producing the deletion scores at
    # the pruning blocks (its cost included, as the paper's timing does)
    asecs, _ = timed(lambda i: forward(sets[i % nsets], True, with_actor=True), args.steps,
                     max(args.warmup, 3))
    ast = max(P.dora_read_status(P.dora_workspace_status(L["actor"]["ws"])) for L in lanes)
    result["with_actor"] = {
        "value": round(cfg.batch * args.steps * world / asecs, 1), "unit": UNIT,
        "ms_per_step": round(1000 * asecs / args.steps, 4),
        "actor_ms_per_step": round(1000 * (asecs - secs) / args.steps, 4),
        "device_status": ast,
        "what": "actor at random init (gate, width-128 encoder, budget head, selector) on each "
                "pruning block's keys; its scores choose the deleted tokens, the configured keep "
                "counts stay"}

    # the same pruned step replayed as CUDA graphs (one per input set)
    try:
        graphs = []
        for r in range(nsets):
            forward(sets[r])
            torch.cuda.synchronize()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                forward(sets[r])
            graphs.append(g)
        gsecs, _ = timed(lambda i: graphs[i % nsets].replay(), args.steps, max(args.warmup, 3))
        result["graph"] = {"value": round(cfg.batch * args.steps * world / gsecs, 1),
                           "unit": UNIT, "ms_per_step": round(1000 * gsecs / args.steps, 4)}
        del graphs
    except Exception as e:                       # context figure only
        result["graph"] = {"unavailable": f"{type(e).__name__}: {e}"[:200]}

    # the complete online forward (App. E.4): patch embedding from the images,
    # the blocks (the actor choosing the deleted tokens at the pruning
    # blocks), and the classifier head; and the same unpruned, for DORA/Native
    if split == 1:
        eh = S.embed_head_weights(cfg, args.seed)
        E = {k: bf(v) for k, v in eh.items()}
        lc1 = cfg.readout == "lc1"                 # DINOv2: [LN CLS, mean LN visual] features
        head = P.dora_classifier_head_lc1 if lc1 else P.dora_classifier_head
        w_head = torch.zeros(1024, E["w_head"].shape[1], dtype=torch.bfloat16, device=dev)
        w_head[:1000] = E["w_head"]
        b_head = torch.zeros(1024, dtype=torch.bfloat16, device=dev)
        b_head[:1000] = E["b_head"]
        imgs = [bf(S.images_bf16(cfg, args.seed + 7 + r)) for r in range(nsets)]
        side = int(imgs[0].shape[-1])
        x0 = torch.zeros(t_cap, cfg.dim, dtype=torch.bfloat16, device=dev)
        logits = torch.zeros(cfg.batch, 1024, dtype=torch.bfloat16, device=dev)
        ews = P.dora_patch_embed(imgs[0], E["w_pe"], E["b_pe"], E["cls"], E["pos"], cfg.patch,
                                 x0, stream=stream)
        hws = None

        def full_step(i, pruned):
            nonlocal hws
            r = i % nsets
            P.dora_patch_embed(imgs[r], E["w_pe"], E["b_pe"], E["cls"], E["pos"], cfg.patch, x0,
                               ews, stream=stream)
            (xf, cuf), = forward(dict(sets[r], x=x0), pruned, with_actor=pruned)
            hws = head(xf, cuf, E["norm_w"], E["norm_b"], 1e-6, w_head, b_head, logits, hws,
                       stream=stream)

        fsecs, _ = timed(lambda i: full_step(i, True), args.steps, max(args.warmup, 3))
        fdsecs, _ = timed(lambda i: full_step(i, False), args.steps, max(args.warmup, 3))
        lens = hw.lengths_per_block(0)
        sched = dict(zip(cfg.prune_blocks, hw.sets[0]["keeps"]))
        rm = 2 if lc1 else 1
        fl = A.trajectory_flops(cfg.depth, cfg.dim, cfg.mlp_dim, cfg.n_tokens, sched,
                                include_embed_head=True, patch=cfg.patch, readout_mult=rm)
        for l in cfg.prune_blocks:
            fl = fl + A.actor_flops(lens[l][0], cfg.dim, cfg.n_vis0, True)
        fld = A.trajectory_flops(cfg.depth, cfg.dim, cfg.mlp_dim, cfg.n_tokens, {},
                                 include_embed_head=True, patch=cfg.patch, readout_mult=rm)
        result["full_forward"] = {
            "value": round(cfg.batch * args.steps * world / fsecs, 1), "unit": UNIT,
            "ms_per_step": round(1000 * fsecs / args.steps, 4),
            "dense_value": round(cfg.batch * args.steps * world / fdsecs, 1),
            "speedup_vs_dense": round(fdsecs / fsecs, 4),
            "gflops_per_image": round(float(fl.mean()) / 1e9, 3),
            "gflops_per_image_dense": round(float(fld.mean()) / 1e9, 3),
            "what": f"images (device-resident, 3x{side}x{side} bf16) -> patch embedding "
                    f"({cfg.patch}-pixel patches) -> {cfg.depth} blocks "
                    "(actor at the pruning blocks, configured keep counts) -> LayerNorm + "
                    "classifier; dense = the same without deletion or actor"}

        # one training rollout step (App. A.3, App. B.2): the forward with
        # Plackett-Luce sampled deletions at the pruning blocks, the Native
        # forward and the complete-prefix shadows of every pruning block but
        # the last riding in the same packed batch, the classifier on every
        # sequence, the fidelity costs, and the log-probabilities of the
        # sampled orders with their gradients
        from paper_2609_34325_gb300.shadow import ShadowRollout
        sr = ShadowRollout(blocks, cfg.batch, cfg.n_tokens, cfg.prune_blocks, dev)
        grng = np.random.default_rng(args.seed + 31)
        gtabs = [[torch.from_numpy((-np.log(-np.log(grng.random(t.shape)))).astype(np.float32))
                  .to(dev) for t in s_["tables"]] for s_ in hw.sets]
        rem = [[torch.from_numpy((np.asarray(b_) - np.asarray(k_)).astype(np.int32)).to(dev)
                for b_, k_ in zip(s_["befores"], s_["keeps"])] for s_ in hw.sets]
        adv = torch.from_numpy(grng.uniform(-1, 1, cfg.batch).astype(np.float32)).to(dev)
        rem2 = [torch.stack(r_) for r_ in rem]
        rwd = torch.zeros(len(cfg.prune_blocks), cfg.batch, dtype=torch.float32, device=dev)
        L0 = lanes[0]

        def train_step(i):
            r = i % nsets
            xo, cuo, _ = sr.forward(sets[r]["x"], L0["cu0"], L0["ids0"], sets[r]["tables"],
                                    sets[r]["keeps"], gumbel=gtabs[r], removals=rem[r],
                                    stream=stream)
            sr.head_and_costs(xo, cuo, E["norm_w"], E["norm_b"], 1e-6, w_head, b_head, lc1=lc1,
                              stream=stream)
            sr.logprob(rem[r], dlogp=adv, stream=stream)
            sr.rewards(rem2[r], 30.0, rwd, stream=stream)

        tsecs, _ = timed(train_step, args.steps, max(args.warmup, 3))
        sst = int(sr.status.item())
        bst = P.dora_read_status(P.dora_workspace_status(sr.ws))
        result["training_step"] = {
            "value": round(cfg.batch * args.steps * world / tsecs, 1), "unit": UNIT,
            "ms_per_step": round(1000 * tsecs / args.steps, 4),
            "sequences": sr.nseq_out, "device_status": max(sst, bst),
            "what": "rollout with Plackett-Luce sampled deletions (Gumbel-top-k, noise an input) "
                    f"at {'/'.join(map(str, cfg.prune_blocks))}, Native forward and the "
                    "complete-prefix shadows branched after each pruning block but the last, "
                    "all in one packed batch through the same kernels; classifier on every "
                    "sequence, fidelity costs (tau = 3), local rewards (a = 30), "
                    "log-probabilities and their gradients"}

    # context: torch eager dense forward of the same shapes and weights
    # (cuBLAS linears, scaled_dot_product_attention), not this library
    try:
        tsecs, _ = timed(lambda i: torch_dense_forward(torch, cfg, blocks, sets[i % nsets]["x"]),
                         max(3, min(args.steps, 20)), max(args.warmup, 3))
        tsteps = max(3, min(args.steps, 20))
        result["torch_eager_dense"] = {
            "value": round(cfg.batch * tsteps * world / tsecs, 1), "unit": UNIT,
            "ms_per_step": round(1000 * tsecs / tsteps, 4),
            "what": "torch eager, same shapes and weights, no deletion: F.layer_norm, F.linear "
                    "(cuBLAS), F.scaled_dot_product_attention, exact GELU"}
    except Exception as e:
        result["torch_eager_dense"] = {"unavailable": f"{type(e).__name__}: {e}"[:200]}

    # End to end through the C ABI with host buffers: every step copies its
    # inputs from pinned host memory and reads its result (final tokens and
    # boundaries) back.  Uploads and readbacks run on two more streams over
    # E2E_SETS rotating buffer sets, so step i+1's upload and step i's
    # readback overlap step i's compute.  (One copy stream over two sets, the
    # readback of step i queued ahead of the upload of step i+2, left some
    # 20-step runs 10-25% slower than the device-only step on the same box;
    # two streams over three sets did not.)
    pin = [dict(x=torch.from_numpy(s["x"].view(np.int16)).view(torch.bfloat16).pin_memory(),
                keeps=[torch.from_numpy(k.astype(np.int32)).pin_memory() for k in s["keeps"]],
                tables=[torch.from_numpy(t).pin_memory() for t in s["tables"]])
           for s in hw.sets]
    dev_in = [dict(x=torch.empty_like(sets[0]["x"]),
                   keeps=[torch.empty_like(k) for k in sets[0]["keeps"]],
                   tables=[torch.empty_like(t) for t in sets[0]["tables"]]) for _ in range(E2E_SETS)]
    host_out = [torch.empty(t_cap, cfg.dim, dtype=torch.bfloat16).pin_memory()
                for _ in range(E2E_SETS)]
    host_cu = [torch.empty(cfg.batch + split, dtype=torch.int32).pin_memory()
               for _ in range(E2E_SETS)]
    h2d = (pin[0]["x"].numel() * 2 + sum(k.numel() * 4 for k in pin[0]["keeps"])
           + sum(t.numel() * 4 for t in pin[0]["tables"]))
    d2h = host_out[0].numel() * 2 + host_cu[0].numel() * 4
    up_stream = torch.cuda.Stream(device=dev)
    down_stream = torch.cuda.Stream(device=dev)

    def ev():
        return torch.cuda.Event()

    def upload(i, after):
        with torch.cuda.stream(up_stream):
            if after is not None:
                up_stream.wait_event(after)
            src, dst = pin[i % nsets], dev_in[i % E2E_SETS]
            dst["x"].copy_(src["x"], non_blocking=True)
            for a, b in zip(dst["keeps"], src["keeps"]):
                a.copy_(b, non_blocking=True)
            for a, b in zip(dst["tables"], src["tables"]):
                a.copy_(b, non_blocking=True)
            e = ev()
            e.record(up_stream)
        return e

    def run_e2e(steps):
        up = {0: upload(0, None)}
        comp, down = {}, {}
        for i in range(steps):
            if i + 1 < steps:
                # input set (i+1) % E2E_SETS is free once step i+1-E2E_SETS is done
                up[i + 1] = upload(i + 1, comp.get(i + 1 - E2E_SETS))
            stream.wait_event(up[i])
            if i - E2E_SETS in down:
                stream.wait_event(down[i - E2E_SETS])         # its output set read back
            outs = forward(dev_in[i % E2E_SETS], True, pair=i % E2E_SETS)
            comp[i] = ev()
            comp[i].record(stream)
            with torch.cuda.stream(down_stream):
                down_stream.wait_event(comp[i])
                c0 = 0
                for L, (x, cu) in zip(lanes, outs):     # each lane's rows and boundaries
                    host_out[i % E2E_SETS][L["r0"]:L["r1"]].copy_(x, non_blocking=True)
                    host_cu[i % E2E_SETS][c0:c0 + L["nb"] + 1].copy_(cu, non_blocking=True)
                    c0 += L["nb"] + 1
                down[i] = ev()
                down[i].record(down_stream)
        stream.wait_event(down[steps - 1])

    esteps = max(3, min(args.steps, 50))
    run_e2e(3)
    torch.cuda.synchronize()
    barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    up_stream.wait_event(e0)
    down_stream.wait_event(e0)
    run_e2e(esteps)
    e1.record(stream)
    torch.cuda.synchronize()
    barrier()
    esecs = max_over_ranks(e0.elapsed_time(e1) / 1000.0)
    result["e2e"] = {"value": round(cfg.batch * esteps * world / esecs, 1), "unit": UNIT,
                     "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
                     "ms_per_step": round(1000 * esecs / esteps, 4),
                     "copies": "pinned host <-> device on an upload and a readback stream, "
                               f"{E2E_SETS} rotating buffer sets, overlapped with compute"}

    # per-kernel pass: the same step driven kernel by kernel with events
    kern = profile_kernels(torch, P, cfg, hw, sets, blocks, dev, stream, t_cap,
                           steps=max(3, min(args.steps, 20)))
    result.update(roofline_report(kern, peaks, peak_src, args.config))
    return result, hw


def torch_dense_forward(torch, cfg, blocks, x):
    """Dense forward of the same blocks in torch eager ops (context figure)."""
    F = torch.nn.functional
    B, N, D, H = cfg.batch, cfg.n_tokens, cfg.dim, cfg.heads
    h = x.view(B, N, D)
    for blk in blocks:
        w = blk.tensors
        a = F.layer_norm(h, (D,), w["ln1_w"], w["ln1_b"], cfg.ln_eps)
        qkv = F.linear(a, w["w_qkv"], w["b_qkv"]).view(B, N, 3, H, D // H).permute(2, 0, 3, 1, 4)
        o = F.scaled_dot_product_attention(qkv[0], qkv[1], qkv[2])
        h = h + F.linear(o.transpose(1, 2).reshape(B, N, D), w["w_proj"], w["b_proj"])
        m = F.layer_norm(h, (D,), w["ln2_w"], w["ln2_b"], cfg.ln_eps)
        h = h + F.linear(F.gelu(F.linear(m, w["w_fc1"], w["b_fc1"])), w["w_fc2"], w["b_fc2"])
    return h


def profile_kernels(torch, P, cfg, hw, sets, blocks, dev, stream, t_cap, steps):
    """Run the pruned step launch by launch through the fine-grained entry
    points (the same kernels dora_pruned_block launches), bracketing each
    launch with CUDA events on the launching stream.  Returns per-class times
    and algorithmic work.

    One difference: at a pruning block dora_pruned_block merges the kept
    rows' slice moments inside the fused selection and skips the
    projection's merge launch; the public dora_select_compact takes row
    moments, so this pass runs that merge launch (23 merges a DeiT-B step
    against the block's 20) and its selection copies merged moments."""
    d, m = cfg.dim, cfg.mlp_dim
    bf16, f32 = torch.bfloat16, torch.float32
    sm = torch.zeros(d // 64, t_cap, 2, dtype=f32, device=dev)      # slice moments
    mv = torch.zeros(t_cap, 2, dtype=f32, device=dev)               # row moments
    mv2 = torch.zeros(t_cap, 2, dtype=f32, device=dev)              # after a deletion
    mvx = [torch.zeros(t_cap, 2, dtype=f32, device=dev) for _ in range(2)]   # between blocks
    # the folded QKV and fc1 weights, as dora_fold_block_weights makes them
    folded = []
    for blk in blocks:
        w = blk.tensors
        fl = {}
        for name, n_out, g, be, b in (("qkv", 3 * d, "ln1_w", "ln1_b", "b_qkv"),
                                      ("fc1", m, "ln2_w", "ln2_b", "b_fc1")):
            fl[name] = (torch.zeros(n_out, d, dtype=bf16, device=dev),
                        torch.zeros(n_out, dtype=f32, device=dev),
                        torch.zeros(n_out, dtype=f32, device=dev))
            P.dora_fold_ln_linear(w["w_" + name], w[g], w[be], *fl[name], bias=w[b], stream=stream)
        folded.append(fl)
    sb = 8.0 * d / 64          # slice-moment bytes per row
    qkv = torch.zeros(t_cap, 3 * d, dtype=bf16, device=dev)
    o = torch.zeros(t_cap, d, dtype=bf16, device=dev)
    hattn = torch.zeros(t_cap, d, dtype=bf16, device=dev)
    hkeep = torch.zeros(t_cap, d, dtype=bf16, device=dev)
    u = torch.zeros(t_cap, m, dtype=bf16, device=dev)
    xb = [torch.zeros(t_cap, d, dtype=bf16, device=dev) for _ in range(2)]
    cub = [torch.zeros(cfg.batch + 1, dtype=torch.int32, device=dev) for _ in range(2)]
    idb = [torch.zeros(t_cap, dtype=torch.int32, device=dev) for _ in range(2)]
    kept = torch.zeros(t_cap, dtype=torch.int32, device=dev)
    scores = torch.zeros(t_cap, dtype=torch.float32, device=dev)
    cu0 = torch.from_numpy(hw.cu0).to(dev)
    ids0 = torch.from_numpy(hw.ids0).to(dev)
    prune = list(cfg.prune_blocks)
    B = cfg.batch
    records = []   # (class, start_event, end_event, work dict)

    def ev():
        return torch.cuda.Event(enable_timing=True)

    def launch(cls, fn, work):
        a, b = ev(), ev()
        a.record(stream)
        fn()
        b.record(stream)
        records.append((cls, a, b, work))

    for it in range(steps + 1):
        r = it % len(sets)
        inp = sets[r]
        lens = hw.lengths_per_block(r)
        x, cu, ids = inp["x"], cu0, ids0
        if it == 1:
            torch.cuda.synchronize()
            records.clear()
        for l in range(cfg.depth):
            w = blocks[l].tensors
            n_in, n_out = lens[l]
            T, To = int(n_in.sum()), int(n_out.sum())
            rows = cu[B:]
            fl = folded[l]
            mvi = mvx[(l + 1) % 2]                   # the previous block's output moments
            if l == 0:
                launch("row_stats", lambda: P.dora_row_stats(x, mvi, rows_dev=rows,
                                                            stream=stream),
                       dict(bytes=2.0 * T * d + 8.0 * T))
            launch("gemm_qkv", lambda: P.dora_linear_ln(x, mvi, cfg.ln_eps, *fl["qkv"], qkv,
                                                   m_dev=rows, stream=stream),
                   dict(flops=2.0 * T * 3 * d * d, rows=T,
                        bytes=2.0 * (T * d + 3 * d * d + 3 * T * d) + 8.0 * T + 24.0 * d))
            launch("attention", lambda: P.dora_varlen_attn(qkv, cu, cfg.n_tokens, cfg.heads, o,
                                                          stream=stream),
                   dict(flops=A.attention_flops(n_in, cfg.heads), bytes=A.attention_bytes(T, d)))
            out = xb[l % 2]
            launch("gemm_proj",
                   lambda: P.dora_linear_residual_stats(o, w["w_proj"], x, hattn, sm,
                                                        bias=w["b_proj"], m_dev=rows,
                                                        stream=stream),
                   dict(flops=2.0 * T * d * d, rows=T, bytes=2.0 * (3 * T * d + d * d) + sb * T))
            launch("merge_moments", lambda: P.dora_merge_moments(sm, mv, rows_dev=rows,
                                                                stream=stream),
                   dict(bytes=sb * T + 8.0 * T))
            if l in prune:
                j = prune.index(l)
                cuo, ido = cub[j % 2], idb[j % 2]
                launch("gather_scores",
                       lambda: P.dora_gather_scores(inp["tables"][j], ids, cu, scores,
                                                    stream=stream),
                       dict(bytes=12.0 * T))
                # selection fused with the compaction of the kept rows, their
                # ids and row moments: scores, boundaries and keep counts read,
                # kept rows read and written, ids and moments read and
                # written, kept_idx and cu_out written
                launch("select_compact",
                       lambda: P.dora_select_compact(scores, cu, inp["keeps"][j], cfg.n_tokens,
                                                     hattn, kept, cuo, hkeep, ids_in=ids,
                                                     ids_out=ido, mv_in=mv, mv_out=mv2,
                                                     stream=stream),
                       dict(bytes=4.0 * T + 4.0 * B + 4.0 * (B + 1) + 2.0 * 2 * To * d
                            + 16.0 * To + 8.0 * To + 4.0 * To + 4.0 * (B + 1)))
                hk, rows2, mvk = hkeep, cuo[B:], mv2
                cu, ids = cuo, ido
            else:
                hk, rows2, mvk = hattn, rows, mv
            launch("gemm_fc1", lambda: P.dora_linear_ln(hk, mvk, cfg.ln_eps, *fl["fc1"], u,
                                                   gelu=True, m_dev=rows2, stream=stream),
                   dict(flops=2.0 * To * d * m, rows=To,
                        bytes=2.0 * (To * d + d * m + To * m) + 8.0 * To + 8.0 * m))
            if l + 1 < cfg.depth:
                launch("gemm_fc2",
                       lambda: P.dora_linear_residual_stats(u, w["w_fc2"], hk, out, sm,
                                                            bias=w["b_fc2"], m_dev=rows2,
                                                            stream=stream),
                       dict(flops=2.0 * To * m * d, rows=To,
                            bytes=2.0 * (To * m + m * d + 2 * To * d) + sb * To))
                launch("merge_moments", lambda: P.dora_merge_moments(sm, mvx[l % 2],
                                                                    rows_dev=rows2,
                                                                    stream=stream),
                       dict(bytes=sb * To + 8.0 * To))
            else:
                launch("gemm_fc2", lambda: P.dora_linear(u, w["w_fc2"], out, bias=w["b_fc2"],
                                                    residual=hk, epilogue=P.EPI_BIAS_RESIDUAL,
                                                    m_dev=rows2, stream=stream),
                       dict(flops=2.0 * To * m * d, rows=To,
                            bytes=2.0 * (To * m + m * d + 2 * To * d)))
            x = out
    torch.cuda.synchronize()
    agg = {}
    for cls, a, b, work in records:
        e = agg.setdefault(cls, dict(ms=0.0, launches=0, flops=0.0, bytes=0.0, rows=0.0))
        e["ms"] += a.elapsed_time(b)
        e["launches"] += 1
        e["flops"] += work.get("flops", 0.0)
        e["bytes"] += work.get("bytes", 0.0)
        e["rows"] += work.get("rows", 0.0)
    gemm = dict(ms=0.0, launches=0, flops=0.0, bytes=0.0, rows=0.0)
    for k in [k for k in agg if k.startswith("gemm_")]:
        for f in gemm:
            gemm[f] += agg[k][f]
    total = sum(e["ms"] for e in agg.values())
    agg["gemm"] = gemm
    for k, e in agg.items():
        e["share"] = e["ms"] / total if total else 0.0
        e["ms"] /= steps
        e["launches"] //= steps
        e["flops"] /= steps
        e["bytes"] /= steps
        e["rows"] /= steps
        if e["flops"]:
            e["tflops"] = e["flops"] / (e["ms"] * 1e-3) / 1e12
    return agg


def roofline_report(kern, peaks, peak_src, workload):
    tag = f"of {peak_src}"
    g = kern["gemm"]
    gemm_tf = g["flops"] / (g["ms"] * 1e-3) / 1e12
    src = os.path.join(ROOT, "paper_2609_34325_gb300", "csrc", "gemm_tcgen05.cu")
    per_row = NCU_GEMM_BYTES_PER_ROW.get(sha256_of(src)) if workload == "cfg3" else None
    tr = None
    if per_row is not None:
        tr = round(sum(per_row[k] * kern[k]["rows"] for k in per_row) / g["launches"])
    # the per-kernel pass times each launch on its own over a fraction of a
    # second: the burst peak is its denominator
    out = {"roofline": {"kernel": "gemm_tcgen05 (QKV/proj/fc1/fc2)", "bound": "tensor",
                        "achieved": round(gemm_tf, 1), "peak": peaks["bf16_tflops"],
                        "unit": "TFLOP/s", "frac": round(gemm_tf / peaks["bf16_tflops"], 4),
                        "peak_kind": f"bf16 burst ({tag})",
                        "frac_of_sustained": round(gemm_tf / peaks["bf16_tflops_sustained"], 4),
                        "traffic": tr,
                        "traffic_case": None if tr is None else (
                            "ncu DRAM bytes per row of each linear on the micro-benchmark "
                            "(50432 rows), scaled by this step's row counts"),
                        "algorithmic_bytes_per_launch": round(g["bytes"] / g["launches"]),
                        "share_of_step": round(g["share"], 4)}}
    a = kern["attention"]
    at_tf = a["flops"] / (a["ms"] * 1e-3) / 1e12
    ai = a["flops"] / a["bytes"]
    attain = min(peaks["bf16_tflops"], ai * peaks["hbm_gbs"] / 1e3)
    out["roofline_attention"] = {
        "bound": "tensor", "achieved": round(at_tf, 1), "peak": peaks["bf16_tflops"],
        "unit": "TFLOP/s", "frac": round(at_tf / peaks["bf16_tflops"], 4),
        "peak_kind": f"bf16 burst ({tag})", "arith_intensity": round(ai, 1),
        "attainable_from_hbm": round(attain, 1), "frac_of_attainable": round(at_tf / attain, 4),
        "share_of_step": round(a["share"], 4)}
    c = kern["select_compact"]
    c_gbs = c["bytes"] / (c["ms"] * 1e-3) / 1e9
    tok_src = os.path.join(ROOT, "paper_2609_34325_gb300", "csrc", "token_ops.cu")
    # the captured traffic is the DeiT-B case's; other shapes report none
    ctr = NCU_TRAFFIC_SELECT_COMPACT.get(sha256_of(tok_src)) if workload == "cfg3" else None
    out["roofline_compact"] = {
        "kernel": "select_keep_kernel (selection fused with the compaction of the kept rows, "
                  "their ids and row moments)", "bound": "hbm",
        "achieved": round(c_gbs, 1), "peak": peaks["hbm_gbs"], "unit": "GB/s",
        "frac": round(c_gbs / peaks["hbm_gbs"], 4), "peak_kind": f"HBM copy ({tag})",
        "us_per_launch": round(1000 * c["ms"] / c["launches"], 2),
        "algorithmic_bytes_per_launch": round(c["bytes"] / c["launches"]),
        "traffic": None if ctr is None else ctr["traffic"],
        "traffic_case": None if ctr is None else ctr["case"],
        "share_of_step": round(c["share"], 4)}
    out["kernels"] = {k: {"ms_per_step": round(v["ms"], 4), "launches_per_step": v["launches"],
                          "share": round(v["share"], 4),
                          **({"tflops": round(v["tflops"], 1)} if "tflops" in v else {})}
                      for k, v in sorted(kern.items())}
    return out


# ---------------------------------------------------------------------------
# CPU oracle legs
# ---------------------------------------------------------------------------
def oracle_sample(hw, r, images, blocks_subset=None):
    """Run the fp64 oracle forward on the chosen images of input set r.
    Returns seconds and the number of image-blocks processed."""
    import oracle as O
    cfg = hw.cfg
    s = hw.sets[r]
    rows = np.concatenate([np.arange(hw.cu0[i], hw.cu0[i + 1]) for i in images])
    lcu = np.arange(len(images) + 1, dtype=np.int64) * cfg.n_tokens
    x = O.bf16_to_f64(s["x"][rows])
    ids = hw.ids0[rows]
    layers = range(cfg.depth) if blocks_subset is None else blocks_subset
    sched = {blk: j for j, blk in enumerate(cfg.prune_blocks)}
    wf = {l: O.decode_weights(hw.weights[l]) for l in layers}
    t0 = time.perf_counter()
    cu = lcu
    for l in layers:
        if l in sched:
            j = sched[l]
            table = s["tables"][j][list(images)]
            keep = s["keeps"][j][list(images)]
            sc = O.gather_scores(table, cu, ids)
            res = O.pruned_block(x, cu, ids, wf[l], cfg.heads, cfg.ln_eps, sc, keep)
        else:
            res = O.pruned_block(x, cu, ids, wf[l], cfg.heads, cfg.ln_eps)
        if blocks_subset is None:
            x, cu, ids = res["x_out"], res["cu_out"], res["ids_out"]
    return time.perf_counter() - t0, len(images) * len(list(layers))


def cpu_baseline(hw, n_images):
    cfg = hw.cfg
    cores = len(os.sched_getaffinity(0))
    imgs = list(range(n_images))
    secs, _ = oracle_sample(hw, 0, imgs)
    out = {"value": round(n_images / secs, 4), "unit": UNIT, "cores": cores, "kind": "oracle",
           "sample": f"{n_images} of {cfg.batch} images through all {cfg.depth} blocks "
                     f"(fp64 numpy oracle, BLAS threads = {cores} host cores)",
           "seconds": round(secs, 2)}
    # the same oracle confined to one core (process affinity), one image
    saved = os.sched_getaffinity(0)
    try:
        os.sched_setaffinity(0, {min(saved)})
        s1, _ = oracle_sample(hw, 0, [0])
        out["one_core"] = {"value": round(1.0 / s1, 4), "unit": UNIT, "cores": 1,
                           "sample": f"1 image through all {cfg.depth} blocks", "seconds": round(s1, 2)}
    finally:
        os.sched_setaffinity(0, saved)
    return out


def run_reference(args, rank, world):
    """The reference arm: the fp64 oracle (the paper's method written out
    plainly) on the host cores, on the same workload as the GPU arm.  Each
    step is one image of the batch through all of the workload's blocks,
    with that image's deletions at the pruning blocks (images are
    independent, so one image is a bounded sample of the batch's work)."""
    if world > 1 and rank != 0:
        return None
    cfg = S.get_config(args.config)
    hw = HostWorkload(cfg, args.seed, 1)
    cores = len(os.sched_getaffinity(0))

    def step(i):
        return oracle_sample(hw, 0, [i % cfg.batch])[0]

    for i in range(max(args.warmup, 0)):
        step(i)
    t0 = time.perf_counter()
    for i in range(args.steps):
        step(args.warmup + i)
    secs = time.perf_counter() - t0
    value = args.steps / secs
    sample = (f"each step: 1 image of the {cfg.batch}-image batch through all {cfg.depth} "
              "blocks with its deletions (images in turn); fp64 numpy oracle, BLAS threads = "
              f"{cores} host cores")
    return {"metric": METRIC, "value": round(value, 4), "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(1000 * secs / max(args.steps, 1), 3), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": workload_config(cfg, world, args.input_sets),
            "impl": "reference",
            "cpu_baseline": {"value": round(value, 4), "unit": UNIT, "cores": cores,
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": round(value, 4), "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


def main():
    args = parse_args()
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        res = run_reference(args, rank, world)
        if res is not None:
            print(json.dumps(res), flush=True)
        return
    res, hw = run_gpu(args, rank, world, local_rank)
    if rank == 0:
        if hw is not None:
            res["cpu_baseline"] = cpu_baseline(hw, args.cpu_images)
            keeps = hw.sets[0]["keeps"]
            c = S.compression_from_counts(hw.cfg, keeps, hw.sets[0]["befores"])
            sched = dict(zip(hw.cfg.prune_blocks, keeps))
            fl = A.trajectory_flops(hw.cfg.depth, hw.cfg.dim, hw.cfg.mlp_dim, hw.cfg.n_tokens,
                                    sched)
            dense = A.trajectory_flops(hw.cfg.depth, hw.cfg.dim, hw.cfg.mlp_dim,
                                       hw.cfg.n_tokens, {})
            res["workload_stats"] = {"compression_C_mean": round(float(c.mean()), 4),
                                     "block_gflops_per_image_pruned": round(float(fl.mean()) / 1e9, 3),
                                     "block_gflops_per_image_dense": round(float(dense.mean()) / 1e9, 3)}
        print(json.dumps(res), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
