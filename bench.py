#!/usr/bin/env python3
"""Benchmark of the LayerCheck per-step hot path on GB300.

One step = measure (Eq. 1 over every parameter) -> select (Eq. 2-4 and the
staleness guard, decision read back to the host) -> pack of the persisted
layers' weights and Adam moments (§3.1) with the fused snapshot commit.
Default workload: the Llama-3-8B shape (35 layers, 8.03 B bf16 parameters,
fp32 moments; 32.12 GB of weights + snapshot read per step, far larger than
L2), tau = 1e-3, S_max = 8, with synthetic drift regenerated between steps
(outside the timed hot path).

Prints one JSON line:
  value      measure+pack algorithmic GB/s with everything resident in HBM
             (packed stream into device memory), CUDA events on the
             library's stream, summed over the K timed steps;
  e2e        the same bytes through the public API into the pinned host
             store (device->host copies of the packed layers included),
             host clock from lc_measure to lc_wait_durable;
  roofline   the dominant kernel against the measured HBM copy bandwidth;
  cpu_baseline  the oracle (single thread) on a bounded sample.
`--impl reference` times the oracle alone on a bounded sample per step.
"""
import argparse
import hashlib
import json
import math
import os
import re
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "measure+pack GB/s (% of HBM peak); per-step decision ms at 8B Llama shape"
FALLBACK_HBM_GBS = 6800.0


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="8b",
                    choices=["tiny", "1b", "8b", "8b-tensor", "8b-cadence"])
    ap.add_argument("--tau", type=float, default=None)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--shape-blocks", type=int, default=0,
                    help="keep only the first N transformer blocks (small case for kernel captures)")
    ap.add_argument("--path", choices=["scan", "fused", "graph"], default="scan",
                    help="scan: measure against the snapshot (default); fused: AdamW step with "
                         "the drift read off the update, fp32 master weights; graph: the scan "
                         "step replayed as one captured CUDA graph with no host round trip")
    ap.add_argument("--drift", choices=["snapshot", "accumulate"], default="snapshot",
                    help="scan path: measure against the snapshot of each layer's last persistence "
                         "(default), or against the previous step's weights with R <- W written "
                         "every step (Eq. 1 literally; 6 B/param bf16)")
    ap.add_argument("--copy-engine", choices=["bulk", "threads"], default="bulk",
                    help="bulk: the bulk-copy engine through shared memory when every buffer is "
                         "device memory (default); threads: per-thread 16-byte vector copies")
    ap.add_argument("--files", default=None, metavar="DIR",
                    help="also append every e2e step's persisted versions to the checkpoint "
                         "directory DIR (fsync'd), then time the metadata-driven recovery from it "
                         "(lc_store_load_dir + lc_restore); DIR is removed afterwards")
    ap.add_argument("--copy-trace", default=None, metavar="FILE",
                    help="write every span of the library's copy trace in the e2e loop and the "
                         "restore (per staging chunk: kind, step, bytes, start/end ms) to FILE "
                         "as JSON lines")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the short passes over the other workloads (tiny, 1b, 8b at tau 5e-4 "
                         "and 2e-3, 8b-tensor, 8b-cadence) that the default 8b run adds as `configs`")
    ap.add_argument("--host-store-gb", type=float, default=0.0,
                    help="cap the pinned store of the e2e leg (GB; 0: 1.5 x the full state, at most 60%% of "
                         "the host's available memory per local rank); steps that do not fit then pack "
                         "into device memory and are left out of e2e")
    ap.add_argument("--no-dma-check", action="store_true",
                    help="do not run lc_store_check_dma on the e2e store (by default the pinned "
                         "regions the GPU copies into at under half the median rate are kept out of use)")
    ap.add_argument("--lean", action="store_true",
                    help="no fp32 master weights in the generator (small case for kernel captures)")
    return ap.parse_args()


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def whole_job(nbytes, seconds, world, device):
    """(bytes, seconds) of the whole job: every rank's bytes over the slowest
    rank's time, so that bytes / seconds is the job's rate (weak scaling:
    each rank moves its own bytes).  One rank: the inputs unchanged."""
    if world <= 1:
        return float(nbytes), float(seconds)
    import torch
    import torch.distributed as dist
    tb = torch.tensor([float(nbytes)], dtype=torch.float64, device=device)
    tt = torch.tensor([float(seconds)], dtype=torch.float64, device=device)
    dist.all_reduce(tb)
    dist.all_reduce(tt, op=dist.ReduceOp.MAX)
    return tb.item(), tt.item()


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as fh:
            p = json.load(fh)
        return float(p["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, "fallback"


# ---------------------------------------------------------------------------
# ncu traffic summaries in profiles/ (valid only for the exact kernel source)
# ---------------------------------------------------------------------------

def kernel_source_sha(files):
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, "paper_2609_27193_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


KERNEL_FILES = {"measure": ["lc_measure.cu", "lc_bulk.cuh", "lc_reduce.cuh", "lc_internal.cuh"],
                "measure_threads": ["lc_measure.cu", "lc_bulk.cuh", "lc_reduce.cuh", "lc_internal.cuh"],
                "fused_adamw": ["lc_adamw.cu", "lc_bulk.cuh", "lc_reduce.cuh", "lc_internal.cuh"],
                "fused_adamw_threads": ["lc_adamw.cu", "lc_bulk.cuh", "lc_reduce.cuh", "lc_internal.cuh"],
                "pack": ["lc_copy.cu", "lc_bulk.cuh", "lc_internal.cuh"],
                "pack_threads": ["lc_copy.cu", "lc_bulk.cuh", "lc_internal.cuh"]}


def profiled_traffic(kernel, workload, persisted_bytes=None):
    """DRAM bytes per launch from profiles/<kernel>_<workload>.md, if that
    capture was taken of the current kernel source: a fixed figure for the
    measure, a per-persisted-byte figure scaled to the step for the pack."""
    path = os.path.join(ROOT, "profiles", "%s_%s.md" % (kernel, workload))
    try:
        text = open(path).read()
    except OSError:
        return None, None
    m_sha = re.search(r"source_sha256_16:\s*([0-9a-f]+)", text)
    m_full = re.search(r"dram_bytes_per_full_launch:\s*([0-9.eE+]+)", text)
    m_per = re.search(r"dram_bytes_per_persisted_byte:\s*([0-9.eE+]+)", text)
    if not m_sha or not (m_full or m_per):
        return None, None
    if m_sha.group(1) != kernel_source_sha(KERNEL_FILES[kernel]):
        return None, "stale"
    if m_full:
        return float(m_full.group(1)), os.path.relpath(path, ROOT)
    if persisted_bytes is None:
        return None, None
    return float(m_per.group(1)) * persisted_bytes, os.path.relpath(path, ROOT)


# ---------------------------------------------------------------------------
# clocks during the timed region
# ---------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, smax, power, reasons = [], [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
                power.append(float(parts[3]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax),
                "power_w_max": max(power), "samples": len(sm), "reasons": sorted(reasons)}


# ---------------------------------------------------------------------------
# algorithmic bytes
# ---------------------------------------------------------------------------

# lr, beta1, beta2, eps, weight decay of the fused path (lr as in the paper's runs)
FUSED_HP = (1e-5, 0.9, 0.999, 1e-8, 0.01)


def fused_step_bytes(state):
    """AdamW step per param: read w, m, v (fp32) and the bf16 gradient, write
    w, m, v and the bf16 model copy: 28 B; the drift sums add no traffic."""
    return sum(28 * t.numel for t in state.specs)


def measure_bytes(state, accumulate=False):
    tot = 0
    for k, t in enumerate(state.specs):
        esz = 2 if state.dtypes[k] == "bf16" else 4
        tot += t.numel * esz * (3 if accumulate else 2)
    return tot


def layer_payload_bytes(state, fp32_weights=False):
    """Per layer: W bytes + moment bytes (the payload of its packed block)."""
    out = [0] * state.nlayers
    wb = [0] * state.nlayers
    for k, t in enumerate(state.specs):
        esz = 4 if fp32_weights or state.dtypes[k] != "bf16" else 2
        out[t.layer] += t.numel * esz + (8 * t.numel if state.has_moments[k] else 0)
        wb[t.layer] += t.numel * esz
    return out, wb


def pack_bytes(mask, payload, wbytes, fused_commit=True):
    """Read of W, m, v + write of the packed payload (+ write of R)."""
    tot = 0
    for l, sel in enumerate(mask):
        if sel:
            tot += 2 * payload[l] + (wbytes[l] if fused_commit else 0)
    return tot


# ---------------------------------------------------------------------------
# the oracle on a bounded sample (CPU baseline and reference arm)
# ---------------------------------------------------------------------------

def oracle_sample_inputs(workload, nblocks, use_gpu):
    """Host copies of `nblocks` transformer blocks of the workload shape, one
    synthetic training step after the base state."""
    import numpy as np
    from lc_workloads import gen
    from lc_workloads.configs import WORKLOADS
    from lc_workloads.shapes import ModelShape, TensorSpec
    wl = WORKLOADS[workload if workload in WORKLOADS else "8b"]
    shape = wl.shape()
    blocks = [l for l in range(1, shape.nlayers) if shape.layer_names[l].startswith("block")]
    if not blocks:
        blocks = list(range(shape.nlayers))
    chosen = blocks[:nblocks]
    ts = [TensorSpec(t.name, chosen.index(t.layer), t.numel, t.dtype)
          for t in shape.tensors if t.layer in chosen]
    sub = ModelShape(shape.name + "-sample", 0, 0, 0, 0, 0, 0, 0, False, False, ts,
                     len(chosen), [shape.layer_names[l] for l in chosen])
    dev = "cuda" if use_gpu else "cpu"
    st = gen.SyntheticState(sub, device=dev, seed=wl.seed + 77)
    scales = wl.layer_scales(shape)[chosen]
    st.drift(1, scales)
    host = dict(W=st.host_all("W"), R=st.host_all("R"), m=st.host_all("m"), v=st.host_all("v"))
    meta = dict(tensor_layer=st.tensor_layer, numels=st.numels, nlayers=sub.nlayers,
                dtypes=st.dtypes, has_moments=st.has_moments,
                params=int(sum(st.numels)), layer_names=sub.layer_names)
    del st
    if use_gpu:
        import torch
        torch.cuda.empty_cache()
    return host, meta, float(wl.tau), int(wl.max_staleness)


def oracle_step(host, meta, tau, K, t, pack_every=4):
    """One oracle step over the sample: Eq. 1 for every sampled layer, the
    selection rule, and the pack of one layer in `pack_every` (the ~25%
    persisted fraction of the timed workload).  Returns (bytes, seconds)."""
    import numpy as np
    from oracle import oracle as O
    from oracle.sim import OracleRun
    run = OracleRun(meta["tensor_layer"], meta["numels"], meta["nlayers"], meta["dtypes"],
                    meta["has_moments"])
    run.R = host["R"]
    t0 = time.perf_counter()
    u, _ = run.measure(host["W"])
    mask = run.select(u, tau, K, t)
    forced = np.zeros_like(mask)
    forced[::pack_every] = 1
    stream, _ = run.pack(forced, host["W"], host["m"], host["v"], t)
    dt = time.perf_counter() - t0
    nbytes = 0
    for k in range(len(meta["numels"])):
        esz = 2 if meta["dtypes"][k] == "bf16" else 4
        nbytes += 2 * meta["numels"][k] * esz
    nbytes += 2 * int(stream.size)
    return nbytes, dt


def cpu_baseline(workload, seconds, use_gpu):
    host, meta, tau, K = oracle_sample_inputs(workload, 4, use_gpu)
    total_b, total_t, steps = 0, 0.0, 0
    while total_t < seconds and steps < 20:
        b, dt = oracle_step(host, meta, tau, K, steps + 1)
        total_b += b
        total_t += dt
        steps += 1
    return {"value": total_b / total_t / 1e9, "unit": "GB/s", "cores": 1, "kind": "oracle",
            "sample": "%d oracle steps over %d transformer blocks (%d params) of the %s shape: "
                      "Eq. 1 on every sampled parameter, the selection rule, and the pack of "
                      "1 of every 4 sampled layers; single thread, %.1f s"
                      % (steps, meta["nlayers"], meta["params"], workload, total_t)}


def ref_workload_label(name):
    """The workload as the device arm names it in its config line."""
    from lc_workloads.configs import WORKLOADS
    shape = WORKLOADS[name].shape()
    return "%s (%s, %d layers, %d params)" % (name, shape.name, shape.nlayers, shape.numel)


def reference_arm(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    import torch
    use_gpu = torch.cuda.is_available()
    host, meta, tau, K = oracle_sample_inputs(args.workload, 4, use_gpu)
    for i in range(args.warmup):
        oracle_step(host, meta, tau, K, i + 1)
    bs, ts = 0, []
    for i in range(args.steps):
        b, dt = oracle_step(host, meta, tau, K, args.warmup + i + 1)
        bs += b
        ts.append(dt)
    value = bs / sum(ts) / 1e9
    sample = ("oracle (single thread) per step: Eq. 1 over 4 transformer blocks (%d params) of "
              "the %s shape, the selection rule, pack of 1 of 4 layers" % (meta["params"], args.workload))
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "GB/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * sum(ts) / len(ts), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": ref_workload_label(args.workload), "tau": tau, "max_staleness": K,
                       "sample": "4 transformer blocks per step", "parallelism": "dp1"},
            "cpu_baseline": {"value": value, "unit": "GB/s", "cores": 1, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": "GB/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# ---------------------------------------------------------------------------
# our arm
# ---------------------------------------------------------------------------

def files_recovery(P, lc, path, t_fail, written, write_s):
    """§3.5 recovery from the checkpoint directory the e2e loop appended to:
    the manifest picks each layer's newest version at or before t_fail and
    only those blocks are read (CRC-checked), then lc_restore scatters them.
    The directory's pages are dropped from the page cache first (its own
    files only), so the reads come from the disk."""
    import shutil
    for name in ("manifest.lcm", "blocks.lcb"):
        fd = os.open(os.path.join(path, name), os.O_RDONLY)
        try:
            os.posix_fadvise(fd, 0, 0, os.POSIX_FADV_DONTNEED)
        finally:
            os.close(fd)
    recs, _, _, _ = P.manifest_read(path, verify_blocks=False)
    on_disk = os.path.getsize(os.path.join(path, "blocks.lcb"))
    t0 = time.perf_counter()
    store, steps = lc.load_dir(path, t_fail)
    t1 = time.perf_counter()
    lc.restore(store, t_fail)
    t2 = time.perf_counter()
    loaded = sum(lc.layer_block_bytes(l) for l in range(len(steps)))
    store.close()
    shutil.rmtree(path, ignore_errors=True)
    return {"records": len(recs), "block_bytes_on_disk": on_disk, "persisted_bytes": int(written),
            "persist_GBps_fsync": written / write_s / 1e9 if write_s > 0 else None,
            "load_dir_s": t1 - t0, "load_dir_GBps": loaded / (t1 - t0) / 1e9,
            "restore_s": t2 - t1, "recovery_s": t2 - t0, "recovered_bytes": int(loaded),
            "oldest_version_step": int(min(steps)), "t_fail": int(t_fail)}


def restore_leg(torch, dev, P, lc, store, t, tau, full, trace_file=None):
    """§3.5 restore timed on its own: one step that persists every layer
    (S_max = 0) into the cleared store, then lc_restore of that composite
    (host -> device copies through the staging ring, scatter into W, m, v
    and R), against a plain pinned host -> device copy probe."""
    store.clear()
    lc.measure(t)
    lc.select(tau, 0)
    lc.pack_async(store)
    lc.commit_snapshot()
    lc.wait_durable(t)
    torch.cuda.synchronize()
    lc.trace_copies(True)
    t0 = time.perf_counter()
    lc.restore(store, t)
    t1 = time.perf_counter()
    spans, _ = lc.copy_trace()
    lc.trace_copies(False)
    if trace_file:
        with open(trace_file, "a") as fh:
            for x in spans:
                fh.write(json.dumps(dict(x, loop_step=t)) + "\n")
    h = torch.empty(4 << 30, dtype=torch.uint8, pin_memory=True)
    d = torch.empty(4 << 30, dtype=torch.uint8, device=dev)
    best = 0.0
    for _ in range(3):
        torch.cuda.synchronize()
        a = time.perf_counter()
        d.copy_(h, non_blocking=True)
        torch.cuda.synchronize()
        best = max(best, h.numel() / (time.perf_counter() - a) / 1e9)
    del h, d
    return {"bytes": int(full), "s": t1 - t0, "GBps": full / (t1 - t0) / 1e9, "h2d_link_GBps_measured": best,
            "h2d_trace": span_summary(spans, "h2d"), "scatter_trace": span_summary(spans, "scatter")}


def span_summary(spans, kind):
    """Chunk spans of one kind from the library's copy trace: bytes, the
    time the stream spent on them (busy), the window from the first start to
    the last end, and the chunks' own rates."""
    sp = [x for x in spans if x["kind"] == kind and math.isfinite(x["start_ms"]) and x["end_ms"] > x["start_ms"]]
    if not sp:
        return None
    busy = sum(x["end_ms"] - x["start_ms"] for x in sp)
    window = max(x["end_ms"] for x in sp) - min(x["start_ms"] for x in sp)
    nbytes = sum(x["bytes"] for x in sp)
    rates = sorted(x["bytes"] / ((x["end_ms"] - x["start_ms"]) / 1e3) / 1e9 for x in sp)
    pick = lambda q: rates[min(len(rates) - 1, int(q * len(rates)))]
    return {"chunks": len(sp), "bytes": int(nbytes), "busy_ms": busy, "window_ms": window,
            "idle_ms": max(0.0, window - busy), "busy_GBps": nbytes / (busy / 1e3) / 1e9,
            "window_GBps": nbytes / (window / 1e3) / 1e9 if window > 0 else None,
            "chunk_GBps_min": rates[0], "chunk_GBps_p10": pick(0.1), "chunk_GBps_p50": pick(0.5),
            "chunk_GBps_p90": pick(0.9), "chunk_GBps_max": rates[-1]}


def merge_span_summaries(items):
    """Totals over several steps' summaries of one kind."""
    items = [x for x in items if x]
    if not items:
        return None
    busy = sum(x["busy_ms"] for x in items)
    window = sum(x["window_ms"] for x in items)
    nbytes = sum(x["bytes"] for x in items)
    return {"steps": len(items), "chunks": sum(x["chunks"] for x in items), "bytes": int(nbytes),
            "busy_ms": busy, "window_ms": window, "idle_frac": max(0.0, window - busy) / window if window else None,
            "busy_GBps": nbytes / (busy / 1e3) / 1e9, "window_GBps": nbytes / (window / 1e3) / 1e9,
            "chunk_GBps_p10_min": min(x["chunk_GBps_p10"] for x in items),
            "chunk_GBps_p50_median": statistics.median(x["chunk_GBps_p50"] for x in items),
            "chunk_GBps_p90_max": max(x["chunk_GBps_p90"] for x in items)}


def d2h_link_probe(torch, dev, nbytes=4 << 30):
    """Plain device->pinned-host copy bandwidth measured beside the e2e loop
    (the host link is shared with other jobs on the machine, so it varies)."""
    d = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    h = torch.empty(nbytes, dtype=torch.uint8, pin_memory=True)
    best = 0.0
    for _ in range(3):
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        h.copy_(d, non_blocking=True)
        torch.cuda.synchronize()
        best = max(best, nbytes / (time.perf_counter() - t0) / 1e9)
    del d, h
    return best


def d2h_streams_probe(torch, dev, nbytes=4 << 30, chunk=256 << 20):
    """The same copy split into chunks spread round-robin over 1, 2 and 4
    streams (best of 3 each): whether concurrent copies get more of the
    host link than one."""
    d = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    h = torch.empty(nbytes, dtype=torch.uint8, pin_memory=True)
    out = {}
    for ns in (1, 2, 4):
        streams = [torch.cuda.Stream(device=dev) for _ in range(ns)]
        best = 0.0
        for _ in range(3):
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            for i in range(nbytes // chunk):
                with torch.cuda.stream(streams[i % ns]):
                    h[i * chunk:(i + 1) * chunk].copy_(d[i * chunk:(i + 1) * chunk], non_blocking=True)
            torch.cuda.synchronize()
            best = max(best, nbytes / (time.perf_counter() - t0) / 1e9)
        out[str(ns)] = round(best, 1)
    del d, h
    return out


def config_pass(P, torch, dev, st, units, nunits, tau, K, steps, warmup, scales_for, dst, hbm,
                per_tensor=False, gemm=None, regime_of=None, l2_bytes=128 << 20):
    """One short device-resident pass over a workload: a fresh context whose
    base state is the tensors as they are, then `warmup` untimed and `steps`
    timed steps of drift -> measure -> select -> pack into device memory ->
    fused commit (the headline step), CUDA events on the library's stream.
    units[k] is the selection unit of tensor k; scales_for(i) the drift
    scales of step i (per unit, or per tensor with per_tensor)."""
    import numpy as np
    side = torch.cuda.Stream(device=dev)
    main = torch.cuda.current_stream(dev)
    lc = P.LayerCheck(device=dev.index or 0, stream=side)
    lc.register_layout([P.segment(units[k], st.W[k], st.R[k], st.m[k], st.v[k]) for k in range(len(units))],
                       nunits)
    payload, wbytes = [0] * nunits, [0] * nunits
    mbytes = 0
    for k, spec in enumerate(st.specs):
        esz = 2 if st.dtypes[k] == "bf16" else 4
        payload[units[k]] += spec.numel * esz + (8 * spec.numel if st.has_moments[k] else 0)
        wbytes[units[k]] += spec.numel * esz
        mbytes += 2 * spec.numel * esz
    flush = torch.empty(4 * l2_bytes, dtype=torch.uint8, device=dev) if mbytes < 4 * l2_bytes else None
    recs = []
    for i in range(warmup + steps):
        sc = scales_for(i)
        if per_tensor:
            st.drift(1000 + i, None, tensor_scale=sc)
        else:
            st.drift(1000 + i, sc)
        if flush is not None:
            flush.fill_(i & 0xFF)
        side.wait_stream(main)
        main.synchronize()
        if gemm is not None:
            gs, a, b, c = gemm
            with torch.cuda.stream(gs):
                for _ in range(40):
                    torch.matmul(a, b, out=c)
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
        h0 = time.perf_counter()
        ev[0].record(side)
        lc.measure(i + 1)
        ev[1].record(side)
        mask, u, nbytes = lc.select(tau, K)
        h1 = time.perf_counter()
        ev[2].record(side)
        lc.pack_device(dst)
        lc.commit_snapshot()
        ev[3].record(side)
        if i >= warmup:
            recs.append((ev, h1 - h0, mask, nbytes, i))
        main.wait_stream(side)
    torch.cuda.synchronize()
    lc.close()
    l2_note = "L2 flushed before every step" if flush is not None else "inputs larger than L2"
    del flush
    el = lambda r, a, b: r[0][a].elapsed_time(r[0][b])
    meas = [el(r, 0, 1) for r in recs]
    pack = [el(r, 2, 3) for r in recs]
    step = [el(r, 0, 3) for r in recs]
    pbytes = [sum(2 * payload[l] + wbytes[l] for l in np.flatnonzero(r[2])) for r in recs]
    dec = [1e3 * r[1] for r in recs]
    mean = lambda x: sum(x) / len(x)
    out = {"steps": steps, "warmup": warmup, "tau": tau, "max_staleness": K, "units": nunits,
           "params": int(sum(s.numel for s in st.specs)),
           "value": (mbytes * len(recs) + sum(pbytes)) / (sum(step) / 1e3) / 1e9, "unit": "GB/s",
           "ms_per_step": mean(step), "decision_ms_p50": float(np.median(dec)),
           "decision_ms_p99": float(np.percentile(dec, 99)),
           "measure_ms": mean(meas), "measure_frac": mbytes / (mean(meas) / 1e3) / 1e9 / hbm,
           "pack_ms": mean(pack),
           "pack_frac": (mean(pbytes) / (mean(pack) / 1e3) / 1e9 / hbm) if mean(pack) > 0 else None,
           "selected_fraction": float(np.mean([r[2].mean() for r in recs])),
           "persisted_GB_per_step": mean([r[3] for r in recs]) / 1e9,
           "l2": l2_note}
    if regime_of is not None:
        groups = {}
        for r, ms_, pb in zip(recs, step, pbytes):
            g = groups.setdefault(regime_of(r[4]), {"sel": [], "bytes": [], "ms": [], "dec": []})
            g["sel"].append(float(r[2].mean()))
            g["bytes"].append(r[3])
            g["ms"].append(ms_)
            g["dec"].append(1e3 * r[1])
        out["regimes"] = {n: {"steps": len(g["ms"]), "selected_fraction": mean(g["sel"]),
                              "persisted_GB_per_step": mean(g["bytes"]) / 1e9, "step_ms": mean(g["ms"]),
                              "decision_ms_p50": float(np.median(g["dec"]))} for n, g in groups.items()}
    return out


def config_passes(P, torch, dev, st8, dst, hbm, l2_bytes):
    """The other workloads beside the headline (8b at tau 1e-3): tiny, 1b,
    8b at tau 5e-4 and 2e-3, the 291-unit per-tensor layout, and the
    cadence workload's 200 steps with its matmul loop and drift regimes.
    The 8B passes reuse the headline's tensors, each with a fresh context."""
    from lc_workloads import gen
    from lc_workloads.configs import WORKLOADS, cadence_scales
    out = {}
    w8 = WORKLOADS["8b"]
    s8 = w8.shape()
    sc8 = w8.layer_scales(s8)
    units8 = [t.layer for t in s8.tensors]
    for tau in (5e-4, 2e-3):
        t0 = time.perf_counter()
        out["8b tau=%g" % tau] = config_pass(P, torch, dev, st8, units8, s8.nlayers, tau, w8.max_staleness, 10, 3,
                                             lambda i: sc8, dst, hbm, l2_bytes=l2_bytes)
        out["8b tau=%g" % tau]["wall_s"] = time.perf_counter() - t0
    wt = WORKLOADS["8b-tensor"]
    st_shape = wt.shape()
    sct = wt.layer_scales(st_shape)
    t0 = time.perf_counter()
    out["8b-tensor"] = config_pass(P, torch, dev, st8, list(range(len(st_shape.tensors))), st_shape.nlayers,
                                   wt.tau, wt.max_staleness, 10, 3, lambda i: sct, dst, hbm, per_tensor=True,
                                   l2_bytes=l2_bytes)
    out["8b-tensor"]["wall_s"] = time.perf_counter() - t0
    wc = WORKLOADS["8b-cadence"]
    a = torch.randn(8192, 8192, device=dev, dtype=torch.bfloat16)
    b = torch.randn(8192, 8192, device=dev, dtype=torch.bfloat16)
    gemm = (torch.cuda.Stream(device=dev), a, b, torch.empty_like(a))
    warm = 3
    step_of = lambda i: max(1, i - warm + 1)       # timed steps 1..200
    t0 = time.perf_counter()
    out["8b-cadence"] = config_pass(P, torch, dev, st8, units8, s8.nlayers, wc.tau, wc.max_staleness, 200, warm,
                                    lambda i: cadence_scales(wc, s8, step_of(i))[0], dst, hbm, gemm=gemm,
                                    regime_of=lambda i: cadence_scales(wc, s8, step_of(i))[1],
                                    l2_bytes=l2_bytes)
    out["8b-cadence"]["wall_s"] = time.perf_counter() - t0
    del a, b, gemm
    for name in ("1b", "tiny"):
        wl = WORKLOADS[name]
        sh = wl.shape()
        st = gen.SyntheticState(sh, device=dev, seed=wl.seed)
        sc = wl.layer_scales(sh)
        t0 = time.perf_counter()
        out[name] = config_pass(P, torch, dev, st, [t.layer for t in sh.tensors], sh.nlayers, wl.tau,
                                wl.max_staleness, 10, 3, lambda i: sc, dst, hbm, l2_bytes=l2_bytes)
        out[name]["wall_s"] = time.perf_counter() - t0
        del st
        torch.cuda.empty_cache()
    for name, d in out.items():
        d["workload"] = name
    return out


def load_package():
    import paper_2609_27193_gb300 as P
    try:
        P.library()
    except ImportError:
        from paper_2609_27193_gb300 import build as B
        B.build()
        P.library()
    return P


def run_ours(args):
    import numpy as np
    import torch
    rank, world, local = dist_env()
    torch.cuda.set_device(local)          # before the process group, so NCCL binds this rank's GPU
    dev = torch.device("cuda", local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    P = load_package()
    from lc_workloads import gen
    from lc_workloads import shapes
    from lc_workloads.configs import WORKLOADS, cadence_scales

    wl = WORKLOADS[args.workload]
    shape = wl.shape()
    base_scales = wl.layer_scales(shape)
    if args.shape_blocks > 0:
        shape, keep = shapes.first_blocks(shape, args.shape_blocks)
        base_scales = base_scales[keep]
    tau = float(args.tau if args.tau is not None else wl.tau)
    K = wl.max_staleness
    t_setup = time.perf_counter()
    fused = args.path == "fused"
    st = gen.SyntheticState(shape, device=dev, seed=wl.seed + rank,
                            master=fused or not args.lean, snapshot=not fused)
    side = torch.cuda.Stream(device=dev)
    main = torch.cuda.current_stream(dev)
    grads = grad_bias = None
    if fused:
        # fp32 master weights are the optimizer's parameters; the bf16 W is the
        # model copy the step refreshes; no snapshot is kept
        lc = P.LayerCheck(device=local, stream=side, mode=P.LC_DRIFT_ACCUMULATE,
                          copy_engine=args.copy_engine)
        lc.register_layout([P.segment(t.layer, st.M[k], None, st.m[k], st.v[k])
                            for k, t in enumerate(shape.tensors)], shape.nlayers)
        grads = [torch.empty(t.numel, dtype=torch.bfloat16, device=dev) for t in shape.tensors]
        lc.register_optimizer(grads, st.W)
        # per-layer gradient bias: layers with consistent gradients move faster
        grad_bias = gen.u_shape(shape.nlayers, 2.0, 0.05, 0.3, np.random.default_rng(wl.seed + 7))
    else:
        accumulate = args.drift == "accumulate"
        lc = P.LayerCheck(device=local, stream=side, copy_engine=args.copy_engine,
                          mode=P.LC_DRIFT_ACCUMULATE if accumulate else P.LC_DRIFT_SNAPSHOT)
        lc.register_layout([P.segment(t.layer, st.W[k], st.R[k], st.m[k], st.v[k])
                            for k, t in enumerate(shape.tensors)], shape.nlayers)
    sums = None
    if world > 1:
        sums = torch.zeros(3 * shape.nlayers, dtype=torch.float64, device=dev)
        lc.set_layer_sums_buffer(sums)
    full = sum(lc.layer_block_bytes(l) for l in range(shape.nlayers))
    dst = torch.empty(full, dtype=torch.uint8, device=dev)
    payload, wbytes = layer_payload_bytes(st, fp32_weights=fused)
    mbytes = fused_step_bytes(st) if fused else measure_bytes(st, accumulate=args.drift == "accumulate")
    # the pack writes R <- W only in snapshot mode (accumulate mode's measure wrote it)
    pack_commit = not fused and args.drift == "snapshot"
    gemm = None
    if args.workload == "8b-cadence":
        a = torch.randn(8192, 8192, device=dev, dtype=torch.bfloat16)
        b = torch.randn(8192, 8192, device=dev, dtype=torch.bfloat16)
        gemm = (torch.cuda.Stream(device=dev), a, b, torch.empty_like(a))
    torch.cuda.synchronize()
    setup_s = time.perf_counter() - t_setup

    def scales_for(t):
        if wl.regimes:
            return cadence_scales(wl, shape, t)[0]
        return base_scales

    l2_bytes = torch.cuda.get_device_properties(dev).L2_cache_size if hasattr(
        torch.cuda.get_device_properties(dev), "L2_cache_size") else 128 << 20
    flush = None
    if mbytes < 4 * l2_bytes:
        # inputs would stay L2-resident between steps: overwrite L2 before each one
        flush = torch.empty(4 * l2_bytes, dtype=torch.uint8, device=dev)

    def new_inputs(t):
        if not fused:
            st.drift(t, scales_for(t))
            return
        g = torch.Generator(device=dev)
        for k, spec in enumerate(shape.tensors):
            g.manual_seed(gen.mix_seed(wl.seed, t, k, 5))
            tmp = torch.randn(spec.numel, generator=g, device=dev)
            grads[k].copy_(tmp.add_(float(grad_bias[spec.layer])).mul_(1e-3))
            del tmp

    graph = args.path == "graph"
    overflow = []
    spill_ok = [False]      # e2e: the host store cannot take a full step

    def graph_step(t, ev, h0):
        ev[0].record(side)
        s_t = lc.step_graph_launch()     # the graph numbers its own steps (from 0)
        for e in ev[1:]:
            e.record(side)
        try:
            mask, u, nbytes = lc.step_wait(s_t)
        except P.LCError as err:
            if err.status != 5:
                raise
            overflow.append(t)
            mask, u, nbytes = np.zeros(shape.nlayers, np.uint8), None, 0
        h1 = time.perf_counter()
        main.wait_stream(side)
        return dict(ev=ev, decision_s=h1 - h0, host_s=h1 - h0, mask=mask, nbytes=nbytes)

    def step(t, mode, store=None):
        new_inputs(t)
        if flush is not None:
            flush.fill_(t & 0xFF)
        side.wait_stream(main)
        main.synchronize()          # inputs of this step are ready before the clock starts
        if gemm is not None:
            # training-like load on another stream while the step runs
            gs, a, b, c = gemm
            with torch.cuda.stream(gs):
                for _ in range(40):
                    torch.matmul(a, b, out=c)
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(5)]
        h0 = time.perf_counter()
        if graph:
            return graph_step(t, ev, h0)
        ev[0].record(side)
        if fused:
            lc.adamw_step_measure(t, FUSED_HP[0], FUSED_HP[1], FUSED_HP[2], FUSED_HP[3], FUSED_HP[4])
        else:
            lc.measure(t)
        ev[1].record(side)
        if sums is not None:
            import torch.distributed as dist
            with torch.cuda.stream(side):
                dist.all_reduce(sums)
        mask, u, nbytes = lc.select(tau, K)
        h1 = time.perf_counter()
        ev[2].record(side)
        if mode == "device":
            lc.pack_device(dst)
        else:
            try:
                lc.pack_async(store)
            except P.LCError as err:
                # a store smaller than a full step: this step's layers go to
                # device memory instead, and the step is left out of e2e
                if err.status != 5 or not spill_ok[0]:
                    raise
                lc.pack_device(dst)
                mode = "spilled"
        ev[3].record(side)
        lc.commit_snapshot()
        ev[4].record(side)
        if mode == "store":
            lc.wait_durable(t)
        h2 = time.perf_counter()
        main.wait_stream(side)
        return dict(ev=ev, decision_s=h1 - h0, host_s=h2 - h0, mask=mask, nbytes=nbytes,
                    spilled=mode == "spilled")

    if graph:
        lc.step_graph_create(tau, K, dst)

    # ---- device-resident phase: the `value` --------------------------------
    t = 0
    for _ in range(args.warmup):
        t += 1
        step(t, "device")
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    torch.cuda.synchronize()
    c0 = lc.counters()
    clocks = ClockSampler(local)
    clocks.start()
    wall0 = time.perf_counter()
    recs = []
    for _ in range(args.steps):
        t += 1
        recs.append(step(t, "device"))
        recs[-1]["t"] = t
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    wall = time.perf_counter() - wall0
    clk = clocks.stop()
    c1 = lc.counters()
    ms = lambda r, a, b: r["ev"][a].elapsed_time(r["ev"][b])
    step_ms = [ms(r, 0, 4) for r in recs]
    measure_ms = [ms(r, 0, 1) for r in recs]
    select_ms = [ms(r, 1, 2) for r in recs]
    pack_ms = [ms(r, 2, 3) for r in recs]
    decision_ms = [1e3 * r["decision_s"] for r in recs]
    pbytes = [pack_bytes(r["mask"], payload, wbytes, fused_commit=pack_commit) for r in recs]
    tot_bytes = sum(mbytes + pb for pb in pbytes)
    tot_s = sum(step_ms) / 1e3
    frac_sel = float(np.mean([r["mask"].mean() for r in recs]))
    tot_bytes, tot_s = whole_job(tot_bytes, tot_s, world, dev)
    value = tot_bytes / tot_s / 1e9
    regimes = None
    if wl.regimes:
        # the drift regimes of the cadence workload, each summarised on its own
        # (the last one, "sparse", persists about a tenth of the layers)
        regimes = {}
        for i, r in enumerate(recs):
            name = cadence_scales(wl, shape, r["t"])[1]
            g = regimes.setdefault(name, {"steps": 0, "sel": [], "bytes": [], "step_ms": [], "pack_ms": [],
                                          "decision_ms": []})
            g["steps"] += 1
            g["sel"].append(float(r["mask"].mean()))
            g["bytes"].append(r["nbytes"])
            g["step_ms"].append(step_ms[i])
            g["pack_ms"].append(pack_ms[i])
            g["decision_ms"].append(decision_ms[i])
        regimes = {n: {"steps": g["steps"], "selected_fraction": statistics.mean(g["sel"]),
                       "persisted_GB_per_step": statistics.mean(g["bytes"]) / 1e9,
                       "step_ms": statistics.mean(g["step_ms"]), "pack_ms": statistics.mean(g["pack_ms"]),
                       "decision_ms_p50": statistics.median(g["decision_ms"])}
                   for n, g in regimes.items()}

    hbm, peak_src = peaks()
    meas_gbs = mbytes / (statistics.mean(measure_ms) / 1e3) / 1e9
    pack_gbs = (statistics.mean(pbytes) / (statistics.mean(pack_ms) / 1e3) / 1e9
                if statistics.mean(pack_ms) > 0 else 0.0)
    dominant = "measure" if sum(measure_ms) >= sum(pack_ms) else "pack"
    measure_name = "fused_adamw" if fused else "measure"
    mean_persisted = statistics.mean(r["nbytes"] for r in recs)
    pack_name = "pack" if args.copy_engine == "bulk" else "pack_threads"
    measure_prof = measure_name + ("_threads" if args.copy_engine != "bulk" else "")
    traffic, tsrc = profiled_traffic(measure_prof if dominant == "measure" else pack_name,
                                     args.workload, mean_persisted if dominant == "pack" else None)
    if fused and dominant == "pack":
        traffic, tsrc = None, None       # the pack profile is of bf16 weights
    if args.shape_blocks or args.lean:
        traffic, tsrc = None, None       # the profiles describe the full layout
    achieved = meas_gbs if dominant == "measure" else pack_gbs
    roofline = {"bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s",
                "frac": achieved / hbm, "frac_of_nominal_8000": achieved / 8000.0, "traffic": traffic,
                "kernel": measure_name if dominant == "measure" else "pack",
                "peak_source": peak_src + " hbm_gbs (copy bandwidth)",
                "traffic_source": tsrc,
                "algorithmic_bytes_per_launch": (mbytes if dominant == "measure"
                                                 else statistics.mean(pbytes))}
    kernels = {measure_name: {"ms": statistics.mean(measure_ms), "GBps": meas_gbs,
                           "frac": meas_gbs / hbm, "bytes": mbytes},
               "select_and_readback": {"ms": statistics.mean(select_ms)},
               "pack": {"ms": statistics.mean(pack_ms), "GBps": pack_gbs, "frac": pack_gbs / hbm,
                        "bytes": statistics.mean(pbytes)}}
    if graph:
        # one replay covers measure, select, pack and the decision readback:
        # only the whole step is timed, and its bytes are measure + pack
        g_bytes = mbytes + statistics.mean(pbytes)
        g_gbs = g_bytes / (statistics.mean(step_ms) / 1e3) / 1e9
        kernels = {"graph_step": {"ms": statistics.mean(step_ms), "GBps": g_gbs, "frac": g_gbs / hbm,
                                  "bytes": g_bytes, "launches_per_step": 3}}
        roofline = {"bound": "hbm", "achieved": g_gbs, "peak": hbm, "unit": "GB/s",
                    "frac": g_gbs / hbm, "frac_of_nominal_8000": g_gbs / 8000.0, "traffic": None,
                    "kernel": "graph step (measure, select, pack, commit)",
                    "peak_source": peak_src + " hbm_gbs (copy bandwidth)", "traffic_source": None,
                    "algorithmic_bytes_per_launch": g_bytes}

    # ---- end to end through the pinned host store --------------------------
    e2e = None
    if not args.no_e2e:
        avail = 0
        try:
            with open("/proc/meminfo") as fh:
                for line in fh:
                    if line.startswith("MemAvailable:"):
                        avail = int(line.split()[1]) * 1024
        except OSError:
            pass
        # ranks on one host share its memory: each pins at most its share
        avail //= max(1, int(os.environ.get("LOCAL_WORLD_SIZE", world)))
        dma_check = None
        if graph:
            # the replayed pack writes straight into pinned host memory
            cap = full if avail == 0 else min(full, int(avail * 0.6))
            store = None
            hostdst = torch.empty(cap, dtype=torch.uint8, pin_memory=True)
            lc.step_graph_create(tau, K, hostdst)
        else:
            # half the full state as headroom for regions the DMA check keeps
            # out of use (pinned pages the GPU reaches slowly)
            cap = int(full * 1.5) if avail == 0 else min(int(full * 1.5), int(avail * 0.6))
            if args.host_store_gb > 0:
                cap = min(cap, int(args.host_store_gb * 1e9))
            spill_ok[0] = cap < full
            store = P.Store(lc, capacity_bytes=cap)
            if not args.no_dma_check:
                region = 256 << 20
                tchk = time.perf_counter()
                rates, excluded = store.check_dma(lc, region_bytes=region, min_fraction=0.5, passes=6)
                srt = np.sort(rates)
                dma_check = {"region_bytes": region, "regions": int(rates.size), "passes": 6, "min_fraction": 0.5,
                             "excluded_bytes": int(excluded), "excluded_regions": int(excluded // region),
                             "worst_pass_GBps_median": float(srt[srt.size // 2]),
                             "worst_pass_GBps_p10": float(srt[srt.size // 10]), "worst_pass_GBps_min": float(srt[0]),
                             "avoided_bytes": int(store.info()["avoided_bytes"]),
                             "capacity": int(cap), "s": time.perf_counter() - tchk,
                             # slow regions whose exclusion would leave no room for a
                             # step that persists every layer stay in use
                             "rule": "excluded slowest first while a full step still fits; the slow "
                                     "regions left in use are avoided by steps that fit without them"}
        link = d2h_link_probe(torch, dev)
        e_recs, e_bytes = [], []
        f_bytes, f_s = 0, 0.0
        files_note = None
        if args.files and not graph:
            import shutil
            need = 1.3 * statistics.mean(r["nbytes"] for r in recs) * (max(1, args.warmup) + args.steps)
            os.makedirs(args.files, exist_ok=True)
            free = shutil.disk_usage(args.files).free
            if need + (8 << 30) > free:
                files_note = ("skipped: about %.0f GB would be written, %.0f GB free on %s"
                              % (need / 1e9, free / 1e9, args.files))
        traces = []
        spilled = 0
        for i in range(max(1, args.warmup) + args.steps):
            t += 1
            if store is not None:
                lc.trace_copies(True)
            r = step(t, "store", store)
            if store is not None:
                spans, _ = lc.copy_trace()
                if args.copy_trace:
                    with open(args.copy_trace, "a") as fh:
                        for x in spans:
                            fh.write(json.dumps(dict(x, loop_step=t)) + "\n")
                r["d2h_trace"] = span_summary(spans, "d2h")
                r["gather_trace"] = span_summary(spans, "gather")
            if store is not None and args.files and files_note is None:
                f0 = time.perf_counter()
                f_bytes += store.persist_dir(args.files, sync=True)
                f_s += time.perf_counter() - f0
            if store is not None:
                store.clear()
            if i >= max(1, args.warmup):
                if r.get("spilled"):
                    spilled += 1
                    continue
                e_recs.append(r)
                e_bytes.append(mbytes + pack_bytes(r["mask"], payload, wbytes, fused_commit=pack_commit))
        if store is not None:
            lc.trace_copies(False)
        link_after = d2h_link_probe(torch, dev)
        link_streams = d2h_streams_probe(torch, dev)
        e_s = sum(r["host_s"] for r in e_recs)
        e_tot = float(sum(e_bytes))
        e_tot, e_s = whole_job(e_tot, e_s, world, dev)
        if not e_recs or e_s <= 0.0:
            # every timed step persisted more than the host store holds
            e2e = {"skipped": "every timed step persisted more than the %.1f GB pinned store holds "
                              "(host memory or --host-store-gb)" % (cap / 1e9),
                   "steps_spilled_to_device": spilled, "store_dma_check": dma_check}
            e_recs = None
        d2h = statistics.mean(r["nbytes"] for r in e_recs) if e_recs else 0
        if e_recs:
            e2e = {"value": e_tot / e_s / 1e9, "unit": "GB/s", "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": int(d2h),
                   "ms_per_step": 1e3 * e_s / len(e_recs),
                   # steps whose layers did not fit a store smaller than a full step
                   # (--host-store-gb, or a host without room for one per rank)
                   "steps_spilled_to_device": spilled,
                   "d2h_GBps": d2h / (statistics.mean((r["host_s"] - r["decision_s"]) if not graph
                                                      else r["host_s"] for r in e_recs)) / 1e9,
                   # the host link and host memory are shared with other jobs on the
                   # machine: the same copy has measured 50-193 GB/s minutes apart, so
                   # the link is probed right before and right after the loop
                   "d2h_link_GBps_measured": link,
                   "store_dma_check": dma_check,
                   "d2h_link_GBps_after": link_after,
                   # GB/s by number of concurrent copy streams: the link, not the
                   # number of copy engines in use, sets the rate
                   "d2h_link_GBps_by_streams": link_streams,
                   "steps_d2h_ms": [round(1e3 * ((r["host_s"] - r["decision_s"]) if not graph else r["host_s"]), 3)
                                    for r in e_recs],
                   "steps_d2h_bytes": [int(r["nbytes"]) for r in e_recs],
                   # the library's own per-chunk events: D2H spans on its copy
                   # stream (busy = copying, idle = waiting for a gathered chunk)
                   # and the gathers into the staging slots on the context stream
                   "d2h_trace": merge_span_summaries([r.get("d2h_trace") for r in e_recs]),
                   "gather_trace": merge_span_summaries([r.get("gather_trace") for r in e_recs]),
                   "steps_d2h_busy_GBps": [round(r["d2h_trace"]["busy_GBps"], 1) if r.get("d2h_trace") else None
                                           for r in e_recs],
                   "steps_d2h_idle_ms": [round(r["d2h_trace"]["idle_ms"], 2) if r.get("d2h_trace") else None
                                         for r in e_recs],
                   "note": "weights, snapshot and moments are device-resident training state; the "
                           "step's only host traffic is the decision block and the persisted "
                           "layers copied into %s" % ("pinned host memory by the replayed graph's pack"
                                                      if graph else "the pinned store")}
        if store is not None and cap >= full:
            e2e["restore"] = restore_leg(torch, dev, P, lc, store, t + 1, tau, full,
                                         trace_file=args.copy_trace)
            t += 1
        if store is not None:
            store.close()
        if args.files and not graph:
            e2e["files"] = ({"skipped": files_note} if files_note
                            else files_recovery(P, lc, args.files, t, f_bytes, f_s))

    configs = None
    if (world == 1 and not args.no_configs and args.workload == "8b" and args.path == "scan"
            and args.drift == "snapshot" and not args.shape_blocks and args.tau is None
            and args.copy_engine == "bulk"):
        configs = config_passes(P, torch, dev, st, dst, hbm, l2_bytes)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        del dst
        torch.cuda.empty_cache()
        cpu = cpu_baseline(args.workload, args.cpu_seconds, True)

    line = {
        "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": statistics.mean(step_ms), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": "%s (%s, %d layers, %d params)%s" % (
                       wl.name, shape.name, shape.nlayers, shape.numel,
                       ", fused AdamW step + drift, fp32 master weights, bf16 gradients, "
                       "lr %g" % FUSED_HP[0] if fused else ""),
                   "tau": tau, "max_staleness": K,
                   "l2": ("inputs larger than L2 (%.1f GB %s per step)"
                          % (mbytes / 1e9, "moved by the fused step" if fused else "read by the measure")
                          if flush is None else "L2 flushed before every step (%d MiB written; "
                          "%.1f MB read per measure)" % (flush.numel() >> 20, mbytes / 1e6)),
                   "inputs": ("fp32 master weights, bf16 gradients and model copy, fp32 Adam moments, "
                              "no snapshot; AdamW in fp32, drift sums fp32 with fp64 combine"
                              if fused else "bf16 weights and snapshot, fp32 Adam moments; "
                              "arithmetic fp32 with fp64 combine"),
                   "copy_engine": args.copy_engine,
                   "drift": "accumulate (fused AdamW)" if fused else args.drift,
                   "parallelism": "dp%d" % world},
        "decision_ms_p50": statistics.median(decision_ms),
        "decision_ms_p99": float(np.percentile(decision_ms, 99)),
        "selected_fraction": frac_sel,
        "persisted_bytes_per_step": statistics.mean(r["nbytes"] for r in recs),
        "full_state_bytes": int(full),
        "roofline": roofline, "kernels": kernels, "e2e": e2e, "cpu_baseline": cpu,
        "gpu_launches": int(c1["kernel_launches"] - c0["kernel_launches"]),
        "bulk_copy_launches": int(c1["bulk_copy_launches"] - c0["bulk_copy_launches"]),
        "capacity_overflow_steps": overflow,
        "regimes": regimes,
        # short passes over the other workloads (device-resident, like value)
        "configs": configs,
        "clocks": clk, "timed_wall_s_with_input_generation": wall, "setup_s": setup_s,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    lc.close()
    if world > 1:
        dist.destroy_process_group()
    return 0


def main():
    args = parse_args()
    if args.impl == "reference":
        return reference_arm(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
