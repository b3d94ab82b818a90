"""Benchmark of the CAS-Spec tree-verify step on GB300.

Workload (one "step"): the 32-layer Llama-7B-shaped model (d=4096, 32 heads x 128, SwiGLU 11008,
vocab 32000, bf16 weights N(0, 0.02) from the seeded generator), prefix of 2048 committed slots
(N(0, 1) bf16 stand-in K/V), a 64-node seeded token tree (depth <= 8): tree verify pass (all layers,
LM head, fused argmax) -> greedy acceptance -> KV compaction -> rollback of the prefix to 2048 so
every step sees the same workload.  Weights (13.2 GB) and KV (1.1 GB) exceed the 129 MB L2 many
times over, so no L2 flush is needed between steps.

Output: one JSON line (rank 0).  value = device-timed step latency in microseconds (lower is
better); e2e = the same through the C ABI with host-resident inputs copied in and the accepted
path copied out every step; roofline = the dominant kernel (bf16: the per-layer projection chain
Wo -> gate/up -> down -> next QKV or LM head; int8: the W8A8 gate/up projection) from a separate
kernel-timing pass with CUDA events around each launch; cpu_baseline = the fp64 oracle on a
bounded sample (embedding + 1 of 32 layers + LM head, scaled to 32 layers) on the host cores.

`--impl reference` times the CPU oracle alone (the reference arm) on the same metric.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "7B tree-verify step latency (µs, n=64) and % of 8 TB/s HBM roofline"
SEED = 20251026
FALLBACK_HBM_GBS = 6800.0

# name -> (layers kept of the 7B shape, prefix P, tree nodes n, max depth, max branching, fraction of
#          layers skipped, quant mode, verify (accept + compact) or draft (tree reset))
WORKLOADS = {
    "verify7b": (32, 2048, 64, 8, None, 0.0, 0, True),
    "layer7b": (1, 1024, 32, 6, 4, 0.0, 0, True),
    # two layers at the verify sizes (prefix 2048, 64 nodes): a small case for kernel profiles
    "attn7b": (2, 2048, 64, 8, None, 0.0, 0, True),
    # two W8A8 draft layers (prefix 2048, 8 nodes): a small case for profiling the int8 projections
    "w8a8layer7b": (2, 2048, 8, 8, None, 0.0, 1, False),
    "verify13b": (40, 4096, 64, 8, None, 0.0, 0, True),
    # one cascade round: the 60%-skip W8A8 draft appends the tree level by level, the 40%-skip bf16
    # draft re-checks all 64 nodes, then the full verify, acceptance and compaction
    "cascade13b": (40, 4096, 64, 8, None, 0.0, 0, True),
}
for _n in (1, 2, 4, 8):
    WORKLOADS[f"draft7b-skip50-n{_n}"] = (32, 2048, _n, 8, None, 0.5, 0, False)
    WORKLOADS[f"draft7b-int8-n{_n}"] = (32, 2048, _n, 8, None, 0.0, 1, False)
    WORKLOADS[f"draft7b-skip50-int8-n{_n}"] = (32, 2048, _n, 8, None, 0.5, 1, False)
    WORKLOADS[f"draft7b-w4a4-n{_n}"] = (32, 2048, _n, 8, None, 0.0, 2, False)
FAMILY = {"verify13b": "13b", "cascade13b": "13b"}  # others: 7B shape
CASCADE_SKIP = (0.4, 0.6)  # d1 (bf16) and d2 (W8A8) layer-skip fractions of the 13B cascade


def _shape(layers: int | None = None, family: str = "7b"):
    import synth

    s = synth.LLAMA13B if family == "13b" else synth.LLAMA7B
    return synth.ModelShape(s.n_layers if layers is None else layers, s.d_model, s.n_heads, s.head_dim, s.ffn,
                            s.vocab)


def algorithmic_bytes(shape, n: int, P: int, layers_on: int | None = None, quant: int = 0) -> dict:
    """Bytes the step must move: every active weight once (int8, or 4-bit in W4A4 mode, + fp32 row
    scales when quantised), the prefix K/V of active layers, the tree K/V written once, fp32 logits
    written once (activations are < 0.1% and left out)."""
    L = shape.n_layers if layers_on is None else layers_on
    d, F, V = shape.d_model, shape.ffn, shape.vocab
    per_weight = {0: 2.0, 1: 1.0, 2: 0.5}[quant]
    w = int(L * (4 * d * d + 3 * d * F) * per_weight) + (L * (5 * d + 2 * F) * 4 if quant else 0)
    lm = V * d * 2
    kv_read = L * 2 * P * d * 2
    kv_write = L * 2 * n * d * 2
    logits = n * V * 4
    return {"weights": w, "lm_head": lm, "kv_read": kv_read, "kv_write": kv_write, "logits": logits,
            "total": w + lm + kv_read + kv_write + logits}


def chain_bytes(shape, n: int, layers_on: int) -> int:
    """Mean algorithmic bytes of one per-layer chain launch (bf16 mode): Wo, Wg, Wu, Wd and the next
    active layer's Wqkv (the LM head after the last layer) read once; the attention output read
    (bf16), the residual stream read and written twice (fp32), the SwiGLU output written and read
    (bf16), q written and the new K/V written (bf16), the logits written once (fp32)."""
    d, F, V, L = shape.d_model, shape.ffn, shape.vocab, layers_on
    w = L * (d * d + 3 * F * d) * 2 + (L - 1) * 3 * d * d * 2 + V * d * 2
    act = L * (n * d * 2 + 4 * n * d * 4 + 2 * n * F * 2) + (L - 1) * 3 * n * d * 2 + n * V * 4
    return (w + act) // L


def gateup_bytes(shape, n: int, quant: int = 0) -> int:
    """Wg, Wu read (+ row scales) + activations read + U written (bf16)."""
    d, F = shape.d_model, shape.ffn
    if quant:
        return int(2 * F * d * (0.5 if quant == 2 else 1.0)) + 2 * F * 4 + n * d + n * F * 2
    return 2 * F * d * 2 + n * d * 2 + n * F * 2


def measured_peaks() -> tuple[float, str]:
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def recorded_traffic() -> float | None:
    """DRAM bytes per launch of the per-layer chain kernel from the committed ncu summary, if it was
    taken on the current kernel source (the summary records the source hash)."""
    path = os.path.join(ROOT, "profiles", "chain_7b_verify_n64.md")
    src = os.path.join(ROOT, "paper_2510_26843_gb300", "csrc", "chain.cu")
    try:
        text = open(path).read()
        h = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
        m_hash = re.search(r"source_sha256_16:\s*([0-9a-f]+)", text)
        m_tr = re.search(r"dram_bytes_per_launch:\s*([0-9.eE+]+)", text)
        if m_hash and m_tr and m_hash.group(1) == h:
            return float(m_tr.group(1))
    except OSError:
        pass
    return None


# ------------------------------------------------------------------------------------------------
# clocks during the timed region
# ------------------------------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.path = tempfile.mktemp(prefix="clocks_", suffix=".csv")
        self.proc = None
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "50",
                 "-i", str(gpu_index)], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        self.t0 = self.t1 = None

    def mark(self, start: bool) -> None:
        if start:
            self.t0 = time.time()
        else:
            self.t1 = time.time()

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        time.sleep(0.12)
        self.proc.terminate()
        self.proc.wait()
        rows = []
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                ts = time.mktime(time.strptime(parts[0].split(".")[0], "%Y/%m/%d %H:%M:%S"))
                ts += float("0." + parts[0].split(".")[1]) if "." in parts[0] else 0.0
                rows.append((ts, float(parts[1]), float(parts[2]), parts[3], parts[4:]))
            except (ValueError, IndexError):
                continue
        os.unlink(self.path)
        inside = [r for r in rows if self.t0 - 0.06 <= r[0] <= self.t1 + 0.06]
        if not inside and rows:
            mid = 0.5 * (self.t0 + self.t1)
            inside = sorted(rows, key=lambda r: abs(r[0] - mid))[:3]
        if not inside:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in inside for i, v in enumerate(r[4][1:5]) if v.lower().startswith("active")})
        return {"sm_mhz": float(np.median([r[1] for r in inside])), "sm_max_mhz": max(r[2] for r in inside),
                "reasons": reasons, "samples": len(inside)}


# ------------------------------------------------------------------------------------------------
# CPU oracle sample (the reference arm and the cpu_baseline)
# ------------------------------------------------------------------------------------------------
class OracleSampler:
    """fp64 oracle on the 7B shape truncated to its first layer; one sample runs the verify step with
    that layer on (t1) and the step with no layer (t0: embedding, final norm, LM head); the full
    step is estimated as t0 + 32 * (t1 - t0)."""

    def __init__(self, parent, toks, P: int, n_layers: int, mode: int = 0, family: str = "7b"):
        import oracle
        import synth

        sh = _shape(None, family)
        self.sh1 = synth.ModelShape(1, sh.d_model, sh.n_heads, sh.head_dim, sh.ffn, sh.vocab)
        self.w = oracle.Weights.from_seed(SEED, self.sh1, keep_layers=1)
        for name in ("wqkv", "wo", "wg", "wu", "wd"):
            self.w.f64(name, 0)
        self.w.f64("embed")
        self.w.f64("lm_head")
        self.kv = oracle.KVCache(1, sh.n_heads, sh.head_dim, P + len(toks))
        k = synth.bf16_to_f32(synth.prefix_kv_bf16(SEED, sh, 0, "k", P)).astype(np.float64)
        v = synth.bf16_to_f32(synth.prefix_kv_bf16(SEED, sh, 0, "v", P)).astype(np.float64)
        self.kv.load_prefix(0, k, v)
        self.parent, self.toks = parent, toks
        self.n_layers = n_layers
        self.mode = mode
        if mode:
            for name in ("wqkv", "wo", "wg", "wu", "wd"):
                self.w.intq(name, 0, 7 if mode == 2 else 127)
        self.t0 = None

    def _run(self, on: int) -> float:
        import oracle

        self.kv.reset_tree()
        t = time.perf_counter()
        oracle.tree_step(self.w, self.kv, self.toks, self.parent, skip_mask=np.array([on], np.uint8),
                         quant_mode=self.mode)
        return time.perf_counter() - t

    def sample_us(self) -> float:
        if self.t0 is None:
            self.t0 = self._run(0)
        t1 = self._run(1)
        return (self.t0 + self.n_layers * max(t1 - self.t0, 0.0)) * 1e6


def workload_tree(wl):
    import synth

    layers, P, n, depth, branch, skip, mode, verify = wl
    parent = synth.tree(SEED, n, depth, branch)
    toks = synth.tokens(SEED, n, _shape().vocab)
    return parent, toks


def bfs_levels(parent, toks):
    """The tree reordered by depth (parents first) and the [start, end) node range of each level."""
    n = len(parent)
    depth = [0] * n
    for i in range(1, n):
        depth[i] = depth[parent[i]] + 1
    order = sorted(range(n), key=lambda i: (depth[i], i))
    pos = {old: new for new, old in enumerate(order)}
    par = np.array([-1 if parent[o] < 0 else pos[int(parent[o])] for o in order], dtype=np.int32)
    tk = np.array([toks[o] for o in order], dtype=np.int32)
    levels, start = [], 0
    for d in range(max(depth) + 1):
        cnt = sum(1 for x in depth if x == d)
        levels.append((start, start + cnt))
        start += cnt
    return par, tk, levels


def describe(name: str, wl) -> str:
    layers, P, n, depth, branch, skip, mode, verify = wl
    fam = FAMILY.get(name, "7b")
    d = _shape(None, fam).d_model
    if name.startswith("cascade"):
        return (f"{name}: llama{fam}-shape {layers} layers, d{d}, prefix {P}; one cascade round on a {n}-node tree "
                f"(depth<={depth}): {int(CASCADE_SKIP[1] * 100)}%-skip W8A8 draft level by level, "
                f"{int(CASCADE_SKIP[0] * 100)}%-skip bf16 re-check of all nodes, full verify + accept + compact")
    kind = "tree verify + accept + compact" if verify else "draft step (tree reset after)"
    extra = (f", {int(skip * 100)}% layers skipped" if skip else "") + {0: ", bf16", 1: ", W8A8", 2: ", W4A4"}[mode]
    br = f", branching<={branch}" if branch else ""
    return (f"{name}: llama{fam}-shape {layers} layer(s), d{d}, n={n} nodes (depth<={depth}{br}), prefix {P}{extra}; "
            f"{kind}")


def config_block(args, name, wl, graphs: bool) -> dict:
    layers, P, n, depth, branch, skip, mode, verify = wl
    return {"workload": describe(name, wl), "n_tree": n, "prefix_len": P, "tree_depth_max": depth, "seed": SEED,
            "l2": "no flush: the weights + KV streamed per step exceed the 129 MB L2 many times",
            "parallelism": f"replicas{args.gpus}"}


def oracle_estimate(name, wl, parent, toks, seconds: float, steps: int | None = None) -> tuple[float, str]:
    """The oracle's time for one step (or one cascade round) of workload `name`, from bounded samples:
    embedding + 1 layer + LM head, scaled to the active layers of each tree step involved."""
    layers, P, n, depth, branch, skip, mode, verify = wl
    family = FAMILY.get(name, "7b")
    if name.startswith("cascade"):
        import synth

        par, tk, levels = bfs_levels(parent, toks)
        m1, m2 = synth.skip_masks(SEED, layers, list(CASCADE_SKIP))
        parts = [(tk[a:b], np.where(par[a:b] < a, -1, par[a:b] - a), int(m2.sum()), 1) for (a, b) in levels]
        parts += [(tk, par, int(m1.sum()), 0), (tk, par, layers, 0)]
        total, desc = 0.0, []
        for tks, prt, on, md in parts:
            s = OracleSampler(prt, tks, P, on, md, family)
            total += float(np.mean([s.sample_us() for _ in range(2)]))
        return total, (f"fp64 oracle, each of the round's {len(parts)} tree steps sampled as embedding + 1 layer + "
                       f"LM head and scaled to its active layers (draft levels rooted at the level's first node)")
    layers_on = layers if not skip else int(round(layers * (1 - skip)))
    s = OracleSampler(parent, toks, P, layers_on, mode, family)
    t_start = time.perf_counter()
    vals = []
    limit = steps if steps is not None else 20
    while not vals or (time.perf_counter() - t_start < seconds and len(vals) < limit):
        vals.append(s.sample_us())
    return float(np.mean(vals)), (f"fp64 oracle, {len(vals)} x (embedding + 1 of {layers_on} layers + LM head), "
                                  f"scaled to {layers_on} layers")


def run_reference(args) -> None:
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    wl = WORKLOADS[args.workload]
    parent, toks = workload_tree(wl)
    vals = []
    sample = ""
    t_start = time.perf_counter()
    t_timed = 0.0
    for i in range(args.warmup + args.steps):
        t_i = time.perf_counter()
        v1, sample = oracle_estimate(args.workload, wl, parent, toks, 0.0, 1)
        if i >= args.warmup:
            t_timed += time.perf_counter() - t_i
        vals.append(v1)
    v = float(np.mean(vals[args.warmup:]))
    cores = os.cpu_count()
    # Each "step" here is one bounded sample (embedding + one layer + LM head) scaled to the step's
    # active layers: the line says so, and how long the samples really took.
    honest = {"extrapolated": True, "samples_timed": args.steps, "sample_kind": sample,
              "timed_region_s": round(t_timed, 2), "wall_s": round(time.perf_counter() - t_start, 2)}
    out = {"impl": "reference", "metric": METRIC, "value": round(v, 1), "unit": "us", "n_gpus": args.gpus,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(v / 1e3, 3), "higher_is_better": False,
           "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "config": config_block(args, args.workload, wl, False),
           "cpu_baseline": {"value": round(v, 1), "unit": "us", "cores": cores, "kind": "oracle",
                            "sample": sample, **honest},
           "e2e": {"value": round(v, 1), "unit": "us", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
           **honest}
    print(json.dumps(out), flush=True)


# ------------------------------------------------------------------------------------------------
# the GPU arm
# ------------------------------------------------------------------------------------------------
def max_over_ranks(value: float) -> float:
    """The largest value over the ranks of the default process group (the value itself without one).
    Replicas time the same step independently; the job's step time is the slowest replica's."""
    import torch
    import torch.distributed as dist

    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return value
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([value], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_tokens_per_s(n_tree: int, step_us: float, world: int) -> float:
    """Whole-job tree tokens per second: every replica verifies n_tree tokens per step."""
    return n_tree / (step_us * 1e-6) * world


def run_gpu(args) -> None:
    import torch
    import torch.distributed as dist

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))

    import synth
    import paper_2510_26843_gb300 as cs
    from paper_2510_26843_gb300.workload import DeviceKV, DeviceModel

    cs.load_library()
    wl = WORKLOADS[args.workload]
    layers, P, n, depth, branch, skip, mode, verify = wl
    family = FAMILY.get(args.workload, "7b")
    cascade = args.workload.startswith("cascade")
    sh = _shape(layers, family)
    dm = DeviceModel(sh, SEED, with_int8=bool(mode) or cascade)
    kv = DeviceKV(dm, P + 2 * n + 64)
    kv.load_random_prefix(SEED, P)
    parent, toks = workload_tree(wl)
    mask = synth.skip_masks(SEED, layers, [skip])[0] if skip else None
    layers_on = layers if mask is None else int(mask.sum())
    if cascade:  # the tree in level order; nested draft masks d1 (bf16) and d2 (W8A8)
        parent, toks, levels = bfs_levels(parent, toks)
        m1, m2 = synth.skip_masks(SEED, layers, list(CASCADE_SKIP))
    stream = torch.cuda.current_stream()
    cs.set_stream(dm.h, stream)
    tok_d = torch.tensor(toks, dtype=torch.int32, device="cuda")
    par_d = torch.tensor(parent, dtype=torch.int32, device="cuda")
    logits = torch.empty(n, sh.vocab, dtype=torch.float32, device="cuda")
    acc = torch.zeros(n + 2, dtype=torch.int32, device="cuda")
    graphs = not args.no_graphs
    cs.set_options(dm.h, cs.OPT_PDL | cs.OPT_W4_TC | cs.OPT_W8_TC | (cs.OPT_GRAPHS if graphs else 0))

    def step():
        if cascade:
            for (a, b) in levels:  # d2 drafts one level at a time, appended to the tree
                cs.tree_step(dm.h, kv.h, tok_d[a:], par_d[a:], b - a, m2, 1, None)
            cs.kv_reset_tree(kv.h)
            cs.tree_step(dm.h, kv.h, tok_d, par_d, n, m1, 0, None)  # d1 re-checks every node
            cs.kv_reset_tree(kv.h)
        cs.tree_step(dm.h, kv.h, tok_d, par_d, n, mask, mode, logits)
        if verify:
            cs.accept_greedy(dm.h, None, tok_d, par_d, n, acc)
            cs.kv_compact(kv.h, acc)
            cs.kv_set_prefix(kv.h, P)
        else:
            cs.kv_reset_tree(kv.h)

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()

    for _ in range(max(args.warmup, 3)):
        step()
    barrier()
    st = cs.get_status(dm.h)
    if st != 0:
        raise RuntimeError(f"device status after warm-up: {st} ({cs.status_string(st)})")

    # ---- device-timed region ----
    clocks = ClockSampler(local)
    time.sleep(0.2)
    n0 = cs.launch_count(dm.h)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier()
    clocks.mark(True)
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    barrier()
    clocks.mark(False)
    launches = cs.launch_count(dm.h) - n0
    clk = clocks.stop()
    ms = e0.elapsed_time(e1) / args.steps
    ms = max_over_ranks(ms)
    us = ms * 1e3

    # ---- end to end through the C ABI with host buffers ----
    tok_h = torch.from_numpy(np.asarray(toks, dtype=np.int32)).pin_memory()
    par_h = torch.from_numpy(np.asarray(parent, dtype=np.int32)).pin_memory()
    out_d = acc if verify else logits[:, :1]
    out_h = torch.zeros(out_d.shape, dtype=out_d.dtype).pin_memory()
    barrier()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        tok_d.copy_(tok_h, non_blocking=True)
        par_d.copy_(par_h, non_blocking=True)
        step()
        out_h.copy_(out_d, non_blocking=True)
        stream.synchronize()
    e2e_us = (time.perf_counter() - t0) / args.steps * 1e6
    if verify:
        assert 1 <= int(out_h[0]) <= n

    # ---- per-step spread (each step between its own events) and the step without graphs ----
    k = max(1, min(args.steps, 50))
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(k)]
    barrier()
    for a, b in evs:
        a.record(stream)
        step()
        b.record(stream)
    barrier()
    per = sorted(a.elapsed_time(b) * 1e3 for a, b in evs)
    step_stats = {"samples": k, "p50_us": round(per[len(per) // 2], 1),
                  "p90_us": round(per[min(len(per) - 1, int(0.9 * len(per)))], 1)}
    if graphs:
        cs.set_options(dm.h, cs.OPT_PDL | cs.OPT_W4_TC | cs.OPT_W8_TC)
        for _ in range(3):
            step()
        barrier()
        e0.record(stream)
        for _ in range(k):
            step()
        e1.record(stream)
        barrier()
        step_stats["eager_us"] = round(e0.elapsed_time(e1) / k * 1e3, 1)

    # ---- kernel-timing pass: eager launches bracketed by CUDA events on the launch stream ----
    cs.set_options(dm.h, cs.OPT_PDL | cs.OPT_W4_TC | cs.OPT_W8_TC)
    cs.profile(dm.h, True)
    for _ in range(args.steps):
        if cascade:  # per-kernel figures of the round's verify step (the drafts mix kernel kinds)
            cs.tree_step(dm.h, kv.h, tok_d, par_d, n, mask, mode, logits)
            cs.accept_greedy(dm.h, None, tok_d, par_d, n, acc)
            cs.kv_compact(kv.h, acc)
            cs.kv_set_prefix(kv.h, P)
        else:
            step()
    per_kind = {}
    # bf16 mode: "qkv" is the first layer's QKV chain launch, "gateup" the per-layer chains
    names = ["qkv", "attention", "wo", "gateup", "down", "lm_head", "other"]
    for k, name in enumerate(names):
        tot, cnt = cs.profile_read(dm.h, k)
        per_kind[name] = {"ms_per_step": round(tot / args.steps, 4), "launches_per_step": cnt // max(args.steps, 1),
                          "avg_us": round(tot / max(cnt, 1) * 1e3, 2)}
    cs.profile(dm.h, False)
    st = cs.get_status(dm.h)
    if st != 0:
        raise RuntimeError(f"device status after timing: {st} ({cs.status_string(st)})")

    peak, peak_kind = measured_peaks()
    gu_bytes = gateup_bytes(sh, n, mode) if mode else chain_bytes(sh, n, layers_on)
    gu_avg_s = per_kind["gateup"]["avg_us"] * 1e-6
    achieved = gu_bytes / gu_avg_s / 1e9
    ab = algorithmic_bytes(sh, n, P, layers_on, mode)
    if cascade:  # the round's bytes: every draft level, the re-check and the verify
        ab = dict(ab)
        on1, on2 = int(m1.sum()), int(m2.sum())
        total = ab["total"]
        T = 0
        for (a, b) in levels:
            total += algorithmic_bytes(sh, b - a, P + T, on2, 1)["total"]
            T += b - a
        total += algorithmic_bytes(sh, n, P, on1, 0)["total"]
        ab["total"] = total
    # the quantised drafts' projections run on the tensor cores (gemm_f8_kernel: e4m3 codes for W4A4,
    # int8 codes widened to fp16 for W8A8; the options set above keep both on)
    kern = ((f"gemm_f8_kernel ({'W4A4 e4m3' if mode == 2 else 'W8A8 int8 widened to fp16'} gate/up + SwiGLU)")
            if mode else
            "chain_kernel (Wo + residual, gate/up + SwiGLU, down + residual, next QKV or LM head)")

    out = {
        "metric": METRIC, "value": round(us, 1), "unit": "us", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(ms, 4), "higher_is_better": False, "scaling": "weak",
        "vs_baseline": None, "dtype": {0: "bf16", 1: "int8", 2: "int4"}[mode],
        "data": "synthetic (seeded N(0,0.02) weights, N(0,1) prefix KV)",
        "config": config_block(args, args.workload, wl, graphs),
        "launch": {"cuda_graphs": graphs, "pdl": True},
        "step_roofline": {"algorithmic_bytes": ab["total"],
                          "pct_of_8TBps": round(100 * ab["total"] / (us * 1e-6) / 8e12, 2),
                          "frac_of_hbm_peak": round(ab["total"] / (us * 1e-6) / 1e9 / peak, 4),
                          "tokens_per_s": round(job_tokens_per_s(n, us, world), 1)},
        "roofline": {"kernel": f"{kern}, {args.workload}", "bound": "hbm", "achieved": round(achieved, 1),
                     "peak": peak, "peak_source": "measured (MEASURED_PEAKS.json hbm_gbs)" if peak_kind == "measured"
                     else "fallback", "unit": "GB/s", "frac": round(achieved / peak, 4),
                     "traffic": recorded_traffic() if (args.workload == "verify7b") else None,
                     "algorithmic_bytes_per_launch": gu_bytes},
        "kernels": per_kind,
        "step_stats": step_stats,
        "e2e": {"value": round(e2e_us, 1), "unit": "us", "h2d_bytes_per_step": 2 * n * 4,
                "d2h_bytes_per_step": int(out_d.numel() * out_d.element_size())},
        "gpu_launches": int(launches),
        "clocks": clk,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        t_cpu = time.perf_counter()
        v, sample = oracle_estimate(args.workload, wl, parent, toks, args.cpu_seconds)
        out["cpu_baseline"] = {"value": round(v, 1), "unit": "us", "cores": os.cpu_count(), "kind": "oracle",
                               "sample": sample, "extrapolated": True,
                               "timed_region_s": round(time.perf_counter() - t_cpu, 2)}
    if rank == 0:
        print(json.dumps(out), flush=True)
    kv.close()
    dm.close()
    if world > 1:
        dist.destroy_process_group()


def run_dytc(args) -> None:
    """DyTC speculative rounds (Sec. 4.2: Algorithm 1 with K = 2 candidates and top-P 0.8, Algorithm 2,
    the EMA estimates) on the 7B shape through casspec_dytc_round: a 50%-layer-skip bf16 draft, a W8A8
    draft and the prompt-lookup bottom draft, the full model verifying.  The prompt is 512 seeded
    tokens run through the model, so the cache and the lookup history agree.  Rounds synchronise the
    host (it reads drafted tokens back), so they are timed by wall clock after warm-up; the value is
    committed tokens per second.  Weights are random: acceptance here measures the machinery, not a
    trained model's agreement."""
    import torch

    import synth
    import paper_2510_26843_gb300 as cs
    from paper_2510_26843_gb300.workload import DeviceKV, DeviceModel

    cs.load_library()
    sh = _shape()
    P0, rounds = 512, args.warmup + args.steps
    dm = DeviceModel(sh, SEED, with_int8=True)
    kv = DeviceKV(dm, P0 + 65 * rounds + 192)
    stream = torch.cuda.current_stream()
    cs.set_stream(dm.h, stream)
    cs.set_options(dm.h, cs.OPT_PDL | cs.OPT_W4_TC | cs.OPT_W8_TC)
    prompt = synth.prefix_tokens(SEED, P0, sh.vocab)
    logits = torch.empty(64, sh.vocab, dtype=torch.float32, device="cuda")
    for a in range(0, P0, 64):  # prefill in 64-token chains
        t = torch.tensor(prompt[a:a + 64], dtype=torch.int32, device="cuda")
        p = torch.tensor(synth.chain(64), dtype=torch.int32, device="cuda")
        cs.tree_step(dm.h, kv.h, t, p, 64, None, 0, logits)
        cs.kv_compact(kv.h, torch.tensor([64, *range(64), 0], dtype=torch.int32, device="cuda"))
    out = [int(torch.argmax(logits[63]).item())]
    history = torch.zeros(P0 + 65 * rounds + 4 * cs.MAX_TREE, dtype=torch.int32, device="cuda")
    history[:P0] = torch.tensor(prompt, dtype=torch.int32, device="cuda")
    history[P0] = out[0]
    hist_len = P0 + 1

    mask = synth.skip_masks(SEED, sh.n_layers, [0.5])[0]
    cfg = cs.config(sh.n_layers, sh.d_model, sh.n_heads, sh.head_dim, sh.ffn, sh.vocab)
    full = cs.step_bytes(cfg, None, 0, 64, P0)
    costs = [cs.step_bytes(cfg, mask, 0, 8, P0) / full, cs.step_bytes(cfg, None, 1, 8, P0) / full, 0.02]
    cfgs = [(mask, 0), (None, 1), ("pld", 4)]
    sch = cs.Dytc([0.5, 0.8, 0.3], costs, alpha_dn=0.3, c_dn=0.02, k_max=4, t_min=0.5, m_max=64, topk=2, p_tree=0.8)
    # The latency model (Sec. 4.2) fitted to steps measured here: each neural configuration's draft
    # step and the verify, at several tree sizes, timed with CUDA events on the model's stream and
    # fed to the scheduler per arithmetic class; the fitted costs replace the byte ratios.
    fit_cfg = [(mask, 0, (1, 4, 8)), (None, 1, (1, 4, 8)), (None, 0, (16, 32, 64))]
    measured = []
    for m_, mode, sizes in fit_cfg:
        for nn in sizes:
            t = torch.tensor(synth.tokens(SEED + nn, nn, sh.vocab), dtype=torch.int32, device="cuda")
            p = torch.tensor(synth.tree(SEED + nn, nn, 8), dtype=torch.int32, device="cuda")
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
            for rep in range(4):
                if rep == 3:
                    ev[0].record(stream)
                cs.tree_step(dm.h, kv.h, t, p, nn, m_, mode, logits)
                if rep == 3:
                    ev[1].record(stream)
                cs.kv_reset_tree(kv.h)
            torch.cuda.synchronize()
            b = cs.step_bytes(cfg, m_, mode, nn, P0)
            us_step = ev[0].elapsed_time(ev[1]) * 1e3
            sch.observe(mode, b, us_step)
            measured.append({"mode": mode, "skip": m_ is not None, "n": nn, "bytes": b, "us": round(us_step, 1)})
    fitted_w = sch.fit_costs([0, 1, 0], [cs.step_bytes(cfg, mask, 0, 8, P0), cs.step_bytes(cfg, None, 1, 8, P0), 0.0],
                             full, [0.0, 1.0 / 6e6], [200.0, 1e-5], 20.0)
    sch.set_cost(2, 0.02)  # the prompt lookup moves no weights: its cost stays the fixed small value
    fitted = [sch.cost(c) for c in range(3)]
    work = torch.zeros(cs.DYTC_WORK, dtype=torch.int32, device="cuda")
    dlog = torch.empty(cs.MAX_TREE, sh.vocab, dtype=torch.float32, device="cuda")

    def one_round():
        nonlocal hist_len
        toks, nd = sch.round(dm.h, kv.h, cfgs, out[-1], work, history, hist_len, dev_logits=dlog)
        history[hist_len:hist_len + len(toks)] = torch.tensor(toks, dtype=torch.int32, device="cuda")
        hist_len += len(toks)
        out.extend(toks)
        return len(toks), nd

    for _ in range(args.warmup):
        one_round()
    torch.cuda.synchronize()
    st = cs.get_status(dm.h)
    if st != 0:
        raise RuntimeError(f"device status after warm-up: {st} ({cs.status_string(st)})")
    clocks = ClockSampler(int(os.environ.get("LOCAL_RANK", "0")))
    time.sleep(0.2)
    n0 = cs.launch_count(dm.h)
    committed = drafted = 0
    clocks.mark(True)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        c, nd = one_round()
        committed += c
        drafted += nd
    torch.cuda.synchronize()
    t1 = time.perf_counter()
    clocks.mark(False)
    launches = cs.launch_count(dm.h) - n0
    st = cs.get_status(dm.h)
    if st != 0:
        raise RuntimeError(f"device status after the timed rounds: {st} ({cs.status_string(st)})")
    us = (t1 - t0) * 1e6 / args.steps
    line = {
        "metric": "DyTC speculative rounds, 7B shape: committed tokens per second", "impl": "ours",
        "value": round(committed / (t1 - t0), 1), "unit": "tok/s", "n_gpus": 1, "steps": args.steps,
        "warmup": args.warmup, "higher_is_better": True, "dtype": "bf16 + int8 drafts",
        "data": "synthetic (seeded N(0,0.02) weights, seeded 512-token prompt)",
        "config": {"workload": "dytc7b: llama7b-shape 32 layers, prompt 512; drafts 50%-skip bf16, W8A8, "
                               "prompt lookup (n <= 4); K = 2, top-P 0.8, k_max 4, m_max 64",
                   "l2": "no flush: every round streams the weights of several steps (GBs)"},
        "us_per_round": round(us, 1), "tokens_per_round": round(committed / args.steps, 3),
        "drafted_per_round": round(drafted / args.steps, 2),
        "alpha": [round(sch.alpha(c), 4) for c in range(3)],
        "costs": {"byte_ratio": [round(c, 4) for c in costs], "fitted": [round(c, 4) for c in fitted],
                  "used": "fitted", "w_bf16": fitted_w[0], "w_w8a8": fitted_w[1], "steps_measured": measured},
        "gpu_launches": int(launches), "clocks": clocks.stop(),
    }
    print(json.dumps(line), flush=True)
    sch.close()
    kv.close()
    dm.close()


def main() -> None:
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-graphs", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--workload", default="verify7b", choices=sorted(WORKLOADS) + ["dytc7b"])
    args = ap.parse_args()
    if args.workload == "dytc7b":
        if args.impl == "reference":
            print(json.dumps({"impl": "reference", "unavailable": "the oracle's 7B-shape DyTC round takes minutes of "
                                                                  "CPU per round"}), flush=True)
        else:
            run_dytc(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
