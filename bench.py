#!/usr/bin/env python3
"""Complete-detection latency of RTCC vs Barrier on the 8-agent stress
workload (704x200 grid, 150k + 20x500 points per agent, max fusion, fp16),
replayed as a 10 Hz frame stream, plus the encoder's tensor-core throughput
and the fusion kernel's bandwidth.

One step = 30 frame periods of a 10 Hz stream (3 s).  In each period the
same seeded arrival trace is replayed in RTCC and in Barrier mode (the order
alternates between periods), for two spreads of the 8 completion times:
lognormal (mu = ln 10 ms, sigma = 0.8; inter-arrival gaps capped at 2 ms) and
zero (all simultaneous, the branches contend for the SMs), each with the
payloads resident in HBM before release and with the payloads in pinned host
memory read on release.  Two more frames per period run on a context whose
launches carry CUDA events around every backbone launch (their live
durations: the roofline); their latency is not sampled.  L2 is flushed (a
512 MiB device write) before every frame.  Latency = host time the detections
are ready (after the rotated NMS, boxes in host memory) minus host time of the
call that delivered the last payload.

After the timed region, untimed legs: the 4-agent uplink sweep (arrivals from
the slot-level uplink, 4 payload loads x {round-robin, max-rate} x 1,000
frames), the 2-agent tiny, 3-agent pp3 and 5-agent attention workloads, the
release-mechanism A/B (zero-copy vs copy-engine H2D), the predicted-vs-
measured gain, per-layer backbone spans and the CPU oracle baseline.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                    [--detail PATH] [--sweep-frames F]

`value` is the RTCC p50 latency (lognormal spread, resident inputs); `e2e`
the same with host inputs.  --impl reference times the CPU oracle on this
workload.  --detail writes every number (per-layer spans included) to a JSON
file; the printed line keeps the summary.
"""
from __future__ import annotations

import argparse
import dataclasses
import json
import os
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import synth  # noqa: E402

METRIC = "complete-detection latency p50/p99 ms RTCC vs barrier; conv TFLOP/s, fusion GB/s"
# dram__bytes_read.sum + dram__bytes_write.sum per k_backbone launch from an
# ncu capture of this build, keyed by the launch's agent count; None until
# captured (and again once the kernel changes)
BACKBONE_TRAFFIC = {8: 542_687_232, 1: 28_923_392}   # profiles/backbone_stress8.md
WORKLOAD = "stress8"
DATA = ("synthetic: seeded uniform + Gaussian-cluster point clouds, He-normal fp32 weights "
        "rounded to fp16, seeded arrival traces (OPV2V and the trained OpenCOOD model are not "
        "available)")
FLUSH_BYTES = 512 << 20
PERIOD_MS = 100.0           # 10 Hz frame stream
PERIODS_PER_STEP = 30
GAP_CAP_MS = 2.0            # > the encoder work one frame can leave queued (see compress_gaps)
SWEEP_GAP_CAP_MS = 1.0      # 4 pp3 branches


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), float(d["bf16_tflops"]), "measured"
    except Exception:
        return 6800.0, 1900.0, "fallback"


def conv_flops(cfg) -> float:
    """Algorithmic FLOPs of one encoder branch's convs and deconvs (2 per MAC)."""
    return sum(fl for _, fl in layer_table(cfg))


def layer_table(cfg):
    """(name, algorithmic FLOPs) of every conv/deconv of one branch, in the
    library's layer order (block convs, then the neck deconvs)."""
    out = []
    w, h, cin = cfg.grid_w, cfg.grid_h, cfg.pfn_ch
    dims = []
    for bi, (n, ch, st) in enumerate(cfg.blocks):
        for li in range(n):
            s = st if li == 0 else 1
            w, h = w // s, h // s
            out.append((f"b{bi}.c{li} 3x3 s{s} {cin}->{ch} @{w}x{h}", 2.0 * w * h * ch * 9 * cin))
            cin = ch
        dims.append((w, h, ch))
    for bi, s in enumerate(cfg.up_strides):
        bw, bh, bc = dims[bi]
        out.append((f"up{bi} deconv k{s} {bc}->{cfg.up_ch} @{bw * s}x{bh * s}",
                    2.0 * (bw * s) * (bh * s) * cfg.up_ch * bc))
    return out


def fusion_bytes(cfg, k_present: int) -> float:
    """Algorithmic bytes of the fusion+head kernel: each present slot read
    once (16-bit), the fp32 head map written once."""
    cells = cfg.feat_w * cfg.feat_h
    return float(k_present * cells * cfg.feat_ch * 2 + cells * 16 * 4)


def pfn_bytes(cfg, n_pillars: int, n_kept: int, n_raw: int) -> float:
    """Bytes the PFN kernel itself moves for one branch: the kept points'
    16-byte records (gathered), the raw point indices of the kept pillars'
    lists, three per-pillar words (count, offset, cell), and per pillar its
    C_p 16-bit channels into the pseudo-image plus two words (cell2pillar,
    kept count).  The rest of the dense pseudo-image keeps its zeros: the
    first pillar kernel clears only the previous pass's cells."""
    return float(n_kept * 16 + n_raw * 4 + n_pillars * (12 + cfg.pfn_ch * 2 + 8))


def compress_gaps(a, cap_ms):
    """Replay times of one arrival trace with every inter-arrival gap
    shortened to at most cap_ms (the first arrival at 0), keeping the order.

    Neither mode's tail changes as long as cap_ms is at least the encoder
    work that can be queued when a gap begins: Barrier holds every branch
    until the last arrival, and under RTCC the GPU has drained before the
    next arrival either way, so the extra idle time is invisible (checked on
    the oracle's timeline in tests/test_bench_model.py)."""
    K = len(a)
    order = sorted(range(K), key=lambda k: (a[k], k))
    t = [0.0] * K
    for j in range(1, K):
        t[order[j]] = t[order[j - 1]] + min(float(a[order[j]] - a[order[j - 1]]), cap_ms)
    return t


def paired_gain(t_b, t_r, n_boot=2000, seed=0):
    """Paired latency gain Barrier - RTCC over traces replayed in both modes
    (index i of both lists is the same arrival trace), with a percentile
    bootstrap 95% confidence interval of its mean (Sec. V-A-4's paired gain,
    resampled pairs, seeded)."""
    g = np.asarray(t_b, dtype=np.float64) - np.asarray(t_r, dtype=np.float64)
    if g.size == 0:
        return None
    rng = np.random.default_rng(seed)
    means = g[rng.integers(0, g.size, size=(n_boot, g.size))].mean(axis=1)
    return {"pairs": int(g.size), "mean_ms": float(g.mean()), "median_ms": float(np.median(g)),
            "ci95_ms": [float(np.percentile(means, 2.5)), float(np.percentile(means, 97.5))],
            "positive": int((g > 0).sum()),
            "rel_mean": float(np.mean(g / np.asarray(t_b, dtype=np.float64)))}


def predicted_gain(a, c_enc, c_post):
    """T_B - T_R of one arrival trace on the single-stream timeline of the
    paper's execution model (Eqs. 20-22): RTCC starts each encoder at
    max(a_k, the previous encoder's finish) in (a_k, k) order, Barrier starts
    them back to back at A = max a in index order, and the post-join follows
    the last encoder in both.  (Equal to the pre-arrival encoder work W_pre.)"""
    K = len(a)
    g = 0.0
    for k in sorted(range(K), key=lambda k: (a[k], k)):
        g = max(a[k], g) + c_enc[k]
    t_r = g + c_post
    t_b = max(a) + sum(c_enc) + c_post
    return t_b - t_r


def max_over_ranks(vals, dist, device):
    """Element-wise maximum of a few floats over all ranks: with one replica
    per GPU, the job's latency is the worst replica's (and its wall time the
    slowest rank's)."""
    import torch
    t = torch.tensor([float(v) for v in vals], device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(x) for x in t]


def _json_num(o):
    """numpy scalars in the JSON line become plain numbers."""
    return o.item() if hasattr(o, "item") else str(o)


def pct(x, q):
    return float(np.percentile(np.asarray(x, dtype=np.float64), q)) if len(x) else None


def sig(x, n=4):
    """x rounded to n significant digits (None passes through)."""
    if x is None:
        return None
    return float(f"{float(x):.{n}g}")


def quad(r, b):
    """[RTCC p50, RTCC p99, Barrier p50, Barrier p99] in ms, 4 digits."""
    return [sig(pct(r, 50)), sig(pct(r, 99)), sig(pct(b, 50)), sig(pct(b, 99))]


# --------------------------------------------------------------------------
# clocks during the timed region
# --------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.rows = []
        self.proc = None
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) >= 8:
                self.rows.append(parts)

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
        if self.thread is not None:
            self.thread.join(timeout=2)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in self.rows:
            try:
                sm.append(float(r[0]))
                mx.append(float(r[1]))
            except ValueError:
                continue
            for n, v in zip(names, r[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": float(max(mx)),
                "reasons": sorted(reasons), "samples": len(sm)}


# --------------------------------------------------------------------------
# CPU oracle timing (cpu_baseline leg and the reference arm)
# --------------------------------------------------------------------------

def oracle_step(cfg, w, pts_agent, arrivals_list):
    """Time one oracle encoder branch and one oracle post-join; return the
    measured service times and the RTCC tail latency of each arrival trace
    under the single-stream timeline (Eqs. 20-22) with those times."""
    from oracle import forward as of
    from oracle import schedule as sch
    t0 = time.perf_counter()
    enc = of.encoder(pts_agent, w, cfg, store=cfg.dtype)
    t1 = time.perf_counter()
    feats = [enc["feat"]] * cfg.n_agents
    F = of.fuse_max(feats) if cfg.fusion == "max" else of.fuse_attn(feats)
    hd = of.head(F, of.store_round(w["head.w"], cfg.dtype), of.store_round(w["head.b"], cfg.dtype))
    of.detect(hd, cfg)
    t2 = time.perf_counter()
    c_enc = int((t1 - t0) * 1e9)
    c_post = int((t2 - t1) * 1e9)
    tails = []
    for a in arrivals_list:
        a_ns = [int(x * 1e6) for x in a]
        tails.append(sch.simulate(a_ns, [c_enc] * cfg.n_agents, [c_post], "rtcc")["T_tail"] / 1e6)
    return c_enc / 1e6, c_post / 1e6, tails


def _workload_desc(cfg):
    return (f"{cfg.name}: {cfg.n_agents}-agent PointPillars intermediate fusion, "
            f"{cfg.grid_w}x{cfg.grid_h} pillar grid (0.4 m), {cfg.n_uniform} uniform + "
            f"{cfg.n_clusters}x{cfg.cluster_pts} clustered points per agent, P_max "
            f"{cfg.max_pillars}, N_max {cfg.max_pts}, backbone 3/5/5 convs 64/128/256 ch, "
            f"deconv neck to {cfg.feat_w}x{cfg.feat_h}x{cfg.feat_ch}, {cfg.fusion} fusion, "
            f"1x1 head, top-{cfg.max_boxes} decode + rotated NMS; 10 Hz frame stream, arrivals "
            f"lognormal(ln 10 ms, 0.8) with gaps capped at {GAP_CAP_MS:g} ms, and all "
            f"simultaneous")


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    cfg = synth.get_config(WORKLOAD)
    w = synth.weights_for(cfg)
    cores = os.cpu_count()
    for s in range(args.warmup):
        oracle_step(cfg, w, synth.points_for(cfg, s, 0), [synth.arrivals_for(cfg, s)])
    tails, c_encs, c_posts = [], [], []
    t_start = time.perf_counter()
    for s in range(args.steps):
        ce, cp, t = oracle_step(cfg, w, synth.points_for(cfg, s, s % cfg.n_agents),
                                [synth.arrivals_for(cfg, s)])
        tails += t
        c_encs.append(ce)
        c_posts.append(cp)
    wall = (time.perf_counter() - t_start) * 1e3
    v = pct(tails, 50)
    sample = (f"per step: one oracle encoder branch (float64 NumPy, {cfg.name} shapes) and one "
              f"{cfg.n_agents}-agent post-join; the frame's RTCC tail for that step's "
              f"lognormal trace from those service times on the single-stream timeline "
              f"(Eqs. 20-22)")
    line = {
        "impl": "reference", "metric": METRIC, "value": v, "unit": "ms", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": wall / max(args.steps, 1),
        "higher_is_better": False, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": DATA, "config": {"workload": _workload_desc(cfg)},
        "latency_ms": {"rtcc_p50": v, "rtcc_p99": pct(tails, 99),
                       "encoder_ms_median": float(np.median(c_encs)),
                       "post_join_ms_median": float(np.median(c_posts))},
        "cpu_baseline": {"value": v, "unit": "ms", "cores": cores, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": v, "unit": "ms", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line, default=_json_num), flush=True)
    return 0


# --------------------------------------------------------------------------
# our arm
# --------------------------------------------------------------------------

class Runner:
    """One library context and the host side of replaying frames on it."""

    _flush = None               # the L2-flush buffer, shared by every runner

    def __init__(self, R, cfg, flags, n_sets=2, frame_base=0):
        import torch
        self.R, self.cfg = R, cfg
        self.K = cfg.n_agents
        self.ctx = R.rtcc_init(R.model_config(cfg, flags=flags),
                               synth.weight_blob(synth.weights_for(cfg)))
        self.sets = [[synth.points_for(cfg, frame_base + f, k) for k in range(self.K)]
                     for f in range(n_sets)]
        self.staging = [R.rtcc_staging_buffer(self.ctx, k) for k in range(self.K)]
        if Runner._flush is None:
            Runner._flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device="cuda")
        self.flush = Runner._flush
        self.fid = 0
        self.staged = -1            # the point set whose payloads are in the device slots
        self.kernels = 0            # kernels the library launched for the frames run so far

    def close(self):
        self.R.rtcc_destroy(self.ctx)

    def frame(self, t, mode, resident, set_idx=0, flush=True, spin=False):
        """Replay one frame: agent k completes at t[k] ms after the start."""
        import torch
        R, c, K = self.R, self.ctx, self.K
        pts = self.sets[set_idx % len(self.sets)]
        if flush:
            self.flush.zero_()
            torch.cuda.synchronize()
        if not resident:
            # the uplink's receiver deposits the payload in pinned host memory
            # (the library's staging buffer); the H2D happens on release,
            # inside the measured span, and leaves the payload in the device
            # slot as well
            for k in range(K):
                self.staging[k][:pts[k].shape[0]] = pts[k]
            if self.staged >= 0:       # the resident path has been set up before
                self.staged = set_idx % len(self.sets)
        elif self.staged != set_idx % len(self.sets):
            for k in range(K):
                assert R.rtcc_stage_resident(c, k, pts[k]) == R.OK
            self.staged = set_idx % len(self.sets)
        assert R.rtcc_set_mode(c, mode) == R.OK
        self.fid += 1
        assert R.rtcc_frame_begin(c, self.fid, 0.0) == R.OK
        t0 = R.rtcc_now_ms() + 0.3
        for k in sorted(range(K), key=lambda k: (t[k], k)):
            due = t0 + t[k]
            while True:
                rem = due - R.rtcc_now_ms()
                if rem <= 0:
                    break
                if rem > 2.0 and not spin:
                    time.sleep((rem - 1.5) / 1e3)
            if resident:
                s = R.rtcc_payload_resident(c, k, float(t[k]))
            else:
                s = R.rtcc_payload_complete(c, k, self.staging[k][:pts[k].shape[0]], float(t[k]))
            assert s == R.OK, R.rtcc_status_str(s)
        s, boxes, _ = R.rtcc_wait_detection(c, 10000)
        assert s == R.OK, R.rtcc_status_str(s)
        info = R.rtcc_get_frame_info(c)
        self.kernels += R.rtcc_kernels_per_frame(c, K)
        nl = min(info.n_backbone_launches, R.MAX_AGENTS)
        return {"tail": info.t_ready_ms - info.t_last_event_ms,
                "launches": [(int(info.backbone_batch[j]), float(info.gpu_launch_ms[j]))
                             for j in range(nl)],
                "fusek": info.gpu_fusion_kernel_ms, "fuse": info.gpu_fusion_ms,
                "pfnk": [info.gpu_pfn_kernel_ms[k] for k in range(K)],
                "n_boxes": len(boxes)}


def replay_leg(R, name, frames, cap_ms, spread=None, flags=0, resident=True, warm=3):
    """RTCC and Barrier tails (ms) of `frames` seeded traces of workload
    `name`, each replayed in both modes (order alternating), payloads resident
    or in pinned host memory, gaps capped at cap_ms (None: as drawn)."""
    cfg = synth.get_config(name)
    if spread == "lognormal":
        cfg = dataclasses.replace(cfg, arrival="lognormal", arrival_args=(float(np.log(10.0)), 0.8))
    run = Runner(R, cfg, flags)
    tails = {R.MODE_RTCC: [], R.MODE_BARRIER: []}
    try:
        for i in range(warm + frames):
            a = synth.arrivals_for(cfg, i, None if spread == "lognormal" else spread)
            t = compress_gaps(a, cap_ms) if cap_ms else [float(x) for x in a]
            for mode in ((R.MODE_RTCC, R.MODE_BARRIER) if i % 2 == 0 else
                         (R.MODE_BARRIER, R.MODE_RTCC)):
                r = run.frame(t, mode, resident, set_idx=i)
                if i >= warm:
                    tails[mode].append(r["tail"])
    finally:
        run.close()
    return tails


def sweep_leg(R, frames, loads=(0.25, 0.5, 1.0, 2.0), t_max=20000, warm=3):
    """The 4-agent uplink sweep on the pp3 network: per frame one channel
    draw (mean SNR U[0, 25] dB per agent, Rayleigh |h|^2 per slot; 1 ms
    slots, one 20 MHz resource block), completion slots from the library's
    slot-level uplink for each payload load (gamma x 16 B x 100k points) and
    scheduler (round-robin, max-rate), gaps capped at 1 ms, each trace
    replayed in RTCC and Barrier mode with resident payloads."""
    cfg = synth.get_config("sweep4")
    K = cfg.n_agents
    bw = 20e6
    scheds = (("rr", R.SCHED_ROUNDROBIN), ("maxrate", R.SCHED_MAXRATE))
    run = Runner(R, cfg, 0)
    cells = {(g, s): {R.MODE_RTCC: [], R.MODE_BARRIER: [], "infeasible": 0, "a_ms": []}
             for g in loads for s, _ in scheds}
    try:
        for f in range(warm + frames):
            d = synth.channel_draws(K, t_max, 1, frame=f, seed=3)
            # per-RB Shannon rate of the Rayleigh-faded link (the workload's
            # channel model): B log2(1 + SNR |h|^2)
            rates = bw * np.log2(1.0 + d["snr"][None, :, None] * d["h2"])
            for g in loads:
                bits = np.full(K, g * 16 * 8 * 100_000, dtype=np.float64)
                for sname, code in scheds:
                    slots, _ = R.rtcc_uplink_simulate(bits, np.ones(K, np.int32), rates, 1e-3, code)
                    cell = cells[(g, sname)]
                    if (slots <= 0).any():
                        if f >= warm:
                            cell["infeasible"] += 1
                        continue
                    a = [float(x) for x in slots]          # ms: a_k = t_k x 1 ms slots
                    t = compress_gaps(a, SWEEP_GAP_CAP_MS)
                    for mode in ((R.MODE_RTCC, R.MODE_BARRIER) if f % 2 == 0 else
                                 (R.MODE_BARRIER, R.MODE_RTCC)):
                        r = run.frame(t, mode, True, set_idx=f, spin=True)
                        if f >= warm:
                            cell[mode].append(r["tail"])
                    if f >= warm:
                        cell["a_ms"].append(max(a))
    finally:
        run.close()
    return cells


def release_ab(R, name, frames=60, spread=None):
    """e2e tails with host payloads: the branch's first kernel reading the
    pinned staging buffer (zero-copy, the default) against a copy-engine H2D
    on a transfer stream gated by a cross-stream event (RTCC_FLAG_H2D_COPY)."""
    out = {}
    for label, flags in (("zero_copy", 0), ("copy_engine", R.FLAG_H2D_COPY)):
        tl = replay_leg(R, name, frames, GAP_CAP_MS, spread=spread, flags=flags, resident=False)
        out[label] = quad(tl[R.MODE_RTCC], tl[R.MODE_BARRIER])
    return out


def layer_spans(R, cfg, flops_tbl, tflops_peak):
    """Per-layer live spans inside the persistent backbone (global-timer
    stamps; RTCC_FLAG_LAYER_TIMES context), for a one-agent launch and for a
    launch over every agent; medians over frames."""
    run = Runner(R, cfg, R.FLAG_LAYER_TIMES)
    out = {}
    try:
        for label, t, mode in (("1", [2.0 * k for k in range(cfg.n_agents)], R.MODE_RTCC),
                               (str(cfg.n_agents), [0.0] * cfg.n_agents, R.MODE_BARRIER)):
            starts, ends = [], []
            for f in range(5):
                run.frame(t, mode, True, set_idx=f)
                if f >= 1:
                    a, e = R.rtcc_get_layer_spans(run.ctx, cfg.n_agents - 1)
                    starts.append(a)
                    ends.append(e)
            st = np.median(np.stack(starts), axis=0)
            en = np.median(np.stack(ends), axis=0)
            nb = int(label)
            rows = []
            for (lname, fl), a_ms, e_ms in zip(flops_tbl, st, en):
                t_ms = float(e_ms - a_ms)
                tf = nb * fl / (t_ms * 1e-3) / 1e12 if t_ms > 0 else 0.0
                rows.append({"layer": lname, "gflop": round(nb * fl / 1e9, 4),
                             "start_us": round(float(a_ms) * 1e3, 2), "us": round(t_ms * 1e3, 2),
                             "tflops": round(tf, 1), "frac": round(tf / tflops_peak, 4)})
            out[label] = {"span_us": round(float(np.max(en)) * 1e3, 1), "rows": rows}
    finally:
        run.close()
    return out


def gain_validation(R, cfg, pairs=35, seed=7):
    """Predicted vs measured gain on resident inputs (Sec. V-C, the 35 paired
    resident-input runs; and the release fidelity of Sec. V-E).

    Service times: each branch's span and the post-join span, from event
    nodes in the graphs of a timeline context (medians over frames whose
    arrivals are 2 ms apart, so branches run alone).  Then `pairs` seeded
    traces with arrivals U[0, S], S = K x the median branch span (so the
    pre-arrival overlap varies from trace to trace), each run in RTCC and in
    Barrier mode on an uninstrumented context without batching (the timeline
    model serialises whole branches); measured gain = Barrier tail - RTCC
    tail.  Lateness = host time a branch's graph was launched minus the host
    time of its modelled release: the call that completed its payload (RTCC),
    or the call that completed the last payload (Barrier).  The controller's
    decision cost is the host time of one rtcc_ctrl_complete through the
    binding (an upper bound: it includes the ctypes call)."""
    K = cfg.n_agents

    def frame(run, mode, a, f):
        t_call = [0.0] * K
        R_ = run.R
        # same replay as Runner.frame, with the host time of each call kept
        pts = run.sets[f % len(run.sets)]
        run.flush.zero_()
        import torch
        torch.cuda.synchronize()
        for k in range(K):
            assert R_.rtcc_stage_resident(run.ctx, k, pts[k]) == R_.OK
        assert R_.rtcc_set_mode(run.ctx, mode) == R_.OK
        run.fid += 1
        assert R_.rtcc_frame_begin(run.ctx, run.fid, 0.0) == R_.OK
        t0 = R_.rtcc_now_ms() + 0.5
        for k in sorted(range(K), key=lambda k: (a[k], k)):
            while R_.rtcc_now_ms() < t0 + a[k]:
                pass
            t_call[k] = R_.rtcc_now_ms()
            assert R_.rtcc_payload_resident(run.ctx, k, float(a[k])) == R_.OK
        s, _, _ = R_.rtcc_wait_detection(run.ctx, 10000)
        assert s == R_.OK
        info = R_.rtcc_get_frame_info(run.ctx)
        last = max(range(K), key=lambda k: (a[k], k))
        late = [info.t_release_ms[k] - (t_call[k] if mode == R_.MODE_RTCC else t_call[last])
                for k in range(K)]
        return (info.t_ready_ms - info.t_last_event_ms, [info.gpu_branch_ms[k] for k in range(K)],
                info.gpu_post_ms, late)

    trun = Runner(R, cfg, R.FLAG_TIMELINE | R.FLAG_NO_BATCH)
    spans, posts = [], []
    for f in range(6):
        _, br, po, _ = frame(trun, R.MODE_RTCC, [2.0 * k for k in range(K)], f)
        if f >= 2:
            spans.append(br)
            posts.append(po)
    trun.close()
    c_enc = [float(x) for x in np.median(np.array(spans), axis=0)]
    c_post = float(np.median(posts))
    spread = K * float(np.median(c_enc))

    run = Runner(R, cfg, R.FLAG_NO_BATCH)
    rng = np.random.default_rng(seed)
    for f in range(3):                                   # warm-up
        frame(run, R.MODE_RTCC, [0.0] * K, f)
    pred, meas, late_r, late_b = [], [], [], []
    for p in range(pairs):
        a = [float(x) for x in rng.uniform(0.0, spread, size=K)]
        modes = (R.MODE_RTCC, R.MODE_BARRIER) if p % 2 == 0 else (R.MODE_BARRIER, R.MODE_RTCC)
        tail = {}
        for m in modes:
            tail[m], _, _, late = frame(run, m, a, p)
            (late_r if m == R.MODE_RTCC else late_b).extend(late)
        meas.append(tail[R.MODE_BARRIER] - tail[R.MODE_RTCC])
        pred.append(predicted_gain(a, c_enc, c_post))
    run.close()

    cc = R.rtcc_ctrl_create(6, 1000)
    dec = []
    for f in range(200):
        R.rtcc_ctrl_begin(cc, f + 1, 0.0)
        for k in range(6):
            t = time.perf_counter()
            R.rtcc_ctrl_complete(cc, k, True, 10, float(k))
            dec.append((time.perf_counter() - t) * 1e6)
        for k in range(6):
            R.rtcc_ctrl_mark(cc, k, R.RUNNING)
            R.rtcc_ctrl_mark(cc, k, R.FINISHED)
        R.rtcc_ctrl_end(cc)
    R.rtcc_ctrl_destroy(cc)

    pred_a, meas_a = np.array(pred), np.array(meas)
    r = float(np.corrcoef(pred_a, meas_a)[0, 1]) if pred_a.std() > 0 and meas_a.std() > 0 else None
    return {"workload": cfg.name, "pairs": pairs,
            "arrivals": f"U[0, {spread:.3f}] ms (K x median branch span), seed {seed}",
            "c_enc_ms": [round(x, 4) for x in c_enc], "c_post_ms": round(c_post, 4),
            "r": r, "mae_ms": float(np.mean(np.abs(pred_a - meas_a))),
            "mean_predicted_ms": float(pred_a.mean()), "mean_measured_ms": float(meas_a.mean()),
            "measured_positive": int((meas_a > 0).sum()),
            "lateness_us": {"rtcc_p50": pct(late_r, 50) * 1e3, "rtcc_p95": pct(late_r, 95) * 1e3,
                            "barrier_p50": pct(late_b, 50) * 1e3,
                            "barrier_p95": pct(late_b, 95) * 1e3},
            "ctrl_decision_us_p50": pct(dec, 50)}


def run_ours(args):
    import torch
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))

    from paper_2608_08330_gb300 import build as B
    if rank == 0 or world == 1:
        B.build()
    if dist is not None:
        dist.barrier()
    B.build()
    from paper_2608_08330_gb300 import rtcc as R
    R.load()

    cfg = synth.get_config(WORKLOAD)
    K = cfg.n_agents
    flops = conv_flops(cfg)
    # latency frames run on a context without instrumentation (the served
    # configuration); two frames per period run on a second context that
    # records CUDA events around every backbone launch and stamps the fusion
    # kernel's span (their latency is not sampled)
    run = Runner(R, cfg, 0)
    trun = Runner(R, cfg, R.FLAG_TIMELINE)
    SPREADS = ("lognormal", "zero")

    def period(p, paced_t0=None):
        """One 100 ms period of the frame stream; returns its records."""
        if paced_t0 is not None:
            due = paced_t0 + p * PERIOD_MS
            rem = due - R.rtcc_now_ms()
            if rem > 0:
                time.sleep(rem / 1e3)
        out = []
        modes = (R.MODE_RTCC, R.MODE_BARRIER) if p % 2 == 0 else (R.MODE_BARRIER, R.MODE_RTCC)
        for spread in SPREADS:
            a = synth.arrivals_for(cfg, p, None if spread == "lognormal" else spread)
            t = compress_gaps(a, GAP_CAP_MS)
            for resident in (True, False):
                for mode in modes:
                    out.append((spread, resident, mode, run.frame(t, mode, resident, set_idx=p)))
        a = compress_gaps(synth.arrivals_for(cfg, p), GAP_CAP_MS)
        out.append(("timeline", True, R.MODE_RTCC, trun.frame(a, R.MODE_RTCC, True, set_idx=p)))
        out.append(("timeline", True, R.MODE_BARRIER,
                    trun.frame([0.0] * K, R.MODE_BARRIER, True, set_idx=p)))
        return out

    for s in range(args.warmup):                     # warm-up steps: the same frames, unpaced
        for p in range(PERIODS_PER_STEP):
            period(100_000 + s * PERIODS_PER_STEP + p)
    k0 = run.kernels + trun.kernels

    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    clocks = ClockSampler(torch.cuda.current_device())
    clocks.start()
    t_start = time.perf_counter()
    t0 = R.rtcc_now_ms() + 1.0
    rec = []
    for s in range(args.steps):
        for p in range(PERIODS_PER_STEP):
            rec += period(s * PERIODS_PER_STEP + p, paced_t0=t0)
    torch.cuda.synchronize()
    wall_ms = (time.perf_counter() - t_start) * 1e3
    if dist is not None:
        dist.barrier()
    clk = clocks.stop()
    n_launch = run.kernels + trun.kernels - k0

    def tails(spread, resident, mode):
        return [r["tail"] for (sp, res, m, r) in rec if sp == spread and res == resident and m == mode]

    lat = {}
    for spread in SPREADS:
        for resident in (True, False):
            key = ("" if resident else "e2e_") + f"{cfg.name}_{spread}"
            lat[key] = quad(tails(spread, resident, R.MODE_RTCC), tails(spread, resident, R.MODE_BARRIER))
    # all-simultaneous RTCC frames whose branches shared one backbone launch
    # (the dispatcher's hold gathered the burst)
    one = [len(r["launches"]) == 1 for (sp, res, m, r) in rec if sp == "zero" and m == R.MODE_RTCC]
    lat["rtcc_zero_one_launch"] = round(sum(one) / len(one), 3) if one else None
    value = pct(tails("lognormal", True, R.MODE_RTCC), 50)
    e2e_value = pct(tails("lognormal", False, R.MODE_RTCC), 50)
    if dist is not None:
        value, e2e_value, wall_ms = max_over_ranks([value, e2e_value, wall_ms], dist, "cuda")
    gain = paired_gain(tails("lognormal", True, R.MODE_BARRIER), tails("lognormal", True, R.MODE_RTCC))

    hbm, tflops_peak, peak_kind = _peaks()
    # backbone launches of the instrumented frames: (agents, ms)
    launches = [x for (sp, res, m, r) in rec if sp == "timeline" for x in r["launches"] if x[1] > 0]
    by_n = {}
    for n, ms in launches:
        by_n.setdefault(n, []).append(ms)
    tot_fl = sum(n * flops for n, _ in launches)
    tot_ms = sum(ms for _, ms in launches)
    enc_tflops = tot_fl / (tot_ms * 1e-3) / 1e12 if tot_ms > 0 else None
    enc_by_n = {str(n): {"launches": len(v), "ms": sig(np.mean(v)),
                         "tflops": sig(n * flops / (np.mean(v) * 1e-3) / 1e12),
                         "frac": sig(n * flops / (np.mean(v) * 1e-3) / 1e12 / tflops_peak, 3)}
                for n, v in sorted(by_n.items())}
    fk_zero = [r["fusek"] for (sp, res, m, r) in rec if sp == "timeline" and m == R.MODE_BARRIER
               and r["fusek"] > 0]
    fu_gbs = fusion_bytes(cfg, K) / (np.mean(fk_zero) * 1e-3) / 1e9 if fk_zero else None
    pf = [t for (sp, res, m, r) in rec if sp == "timeline" for t in r["pfnk"] if t > 0]
    traffic = BACKBONE_TRAFFIC.get(K)

    frames_per_period = 4 * len(SPREADS) + 2
    h2d = sum(int(p.shape[0]) * 16 + 16 for p in run.sets[0]) * 2 * len(SPREADS)   # host frames/period
    d2h = (16 + cfg.max_boxes * 36) * frames_per_period
    line = {
        "metric": METRIC, "value": value, "unit": "ms", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": wall_ms / max(args.steps, 1),
        "higher_is_better": False, "scaling": "weak", "vs_baseline": None, "dtype": "fp16",
        "data": DATA,
        "config": {"workload": _workload_desc(cfg),
                   "step": f"{PERIODS_PER_STEP} periods of a 10 Hz stream; per period "
                           f"{frames_per_period} frames: {{lognormal, zero}} x {{resident, "
                           f"host}} x {{RTCC, Barrier}} + 2 instrumented",
                   "l2": "flushed by a 512 MiB device write before every frame",
                   "inputs": "value: payloads resident in HBM before release; e2e: payloads in "
                             "pinned host memory, read on release inside the measured span",
                   "replicas": world},
        "roofline": {"kernel": "k_backbone (persistent tcgen05 implicit-GEMM backbone: 13 convs + "
                               "3 deconvs of every agent in the launch)",
                     "bound": "tensor", "achieved": sig(enc_tflops), "peak": tflops_peak,
                     "unit": "TFLOP/s",
                     "frac": sig(enc_tflops / tflops_peak, 3) if enc_tflops else None,
                     "peak_kind": f"{peak_kind} bf16 burst (fp16: same nominal rate)",
                     "traffic": traffic, "traffic_launch": f"{K}-agent launch (one-agent: "
                                                           f"{BACKBONE_TRAFFIC.get(1)} B)",
                     "over": "all backbone launches of the instrumented frames, sum of FLOPs / "
                             "sum of CUDA-event durations"},
        "e2e": {"value": e2e_value, "unit": "ms",
                "h2d_bytes_per_step": h2d * PERIODS_PER_STEP,
                "d2h_bytes_per_step": d2h * PERIODS_PER_STEP},
        "clocks": clk,
        "gpu_launches": n_launch,
    }
    detail = {}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        arr = [synth.arrivals_for(cfg, s) for s in range(args.steps * PERIODS_PER_STEP)]
        ce, cp, ct = oracle_step(cfg, synth.weights_for(cfg), run.sets[0][0], arr)
        line["cpu_baseline"] = {
            "value": pct(ct, 50), "unit": "ms", "cores": os.cpu_count(), "kind": "oracle",
            "sample": (f"one oracle encoder branch ({ce:.0f} ms) and one 8-agent post-join "
                       f"({cp:.0f} ms), float64 NumPy; RTCC tail of every timed lognormal trace "
                       f"(uncapped) on the single-stream timeline (Eqs. 20-22)")}
    run.close()
    trun.close()

    if rank == 0:
        legs = {}
        t_leg = time.perf_counter()
        sw = sweep_leg(R, args.sweep_frames)
        sweep = {}
        detail["sweep4"] = {}
        for (g, s), cell in sw.items():
            key = f"{s}{g:g}"
            sweep[key] = quad(cell[R.MODE_RTCC], cell[R.MODE_BARRIER]) + [cell["infeasible"]]
            detail["sweep4"][key] = {
                "quad": sweep[key], "last_arrival_ms_median": sig(pct(cell["a_ms"], 50)),
                "paired_gain": paired_gain(cell[R.MODE_BARRIER], cell[R.MODE_RTCC])}
        legs["sweep_s"] = time.perf_counter() - t_leg
        others = {}
        for name, cap, spread in (("tiny", None, None), ("pp3", GAP_CAP_MS, None),
                                  ("lr5", GAP_CAP_MS, None)):
            tl = replay_leg(R, name, args.leg_frames, cap, spread=spread)
            others[name] = quad(tl[R.MODE_RTCC], tl[R.MODE_BARRIER])
            detail[f"paired_gain_{name}"] = paired_gain(tl[R.MODE_BARRIER], tl[R.MODE_RTCC])
        ab = {"pp3": release_ab(R, "pp3"), cfg.name: release_ab(R, cfg.name)}
        # the paper's placement: block maps fused after the join, neck once
        msc = {}
        for name in ("pp3", "lr5", cfg.name):
            tl = replay_leg(R, name, args.leg_frames // 3, GAP_CAP_MS, flags=R.FLAG_MULTISCALE)
            msc[name] = quad(tl[R.MODE_RTCC], tl[R.MODE_BARRIER])
        detail["multiscale"] = msc
        gv = gain_validation(R, synth.get_config("pp3"))
        detail["gain_validation"] = gv
        detail["layers"] = layer_spans(R, cfg, layer_table(cfg), tflops_peak)
        detail["encoder_by_launch_size"] = enc_by_n
        detail["paired_gain_" + cfg.name] = gain
        detail["release_ab"] = ab
        detail["latency_ms"] = lat
        detail["legs_s"] = legs

        line["latency_ms"] = dict(lat, **others,
                                  quad="[RTCC p50, RTCC p99, Barrier p50, Barrier p99]",
                                  frames_per_mode=len(tails("lognormal", True, R.MODE_RTCC)),
                                  leg_frames=args.leg_frames,
                                  gain=[sig(gain["mean_ms"]), sig(gain["ci95_ms"][0]),
                                        sig(gain["ci95_ms"][1]), gain["positive"]]
                                  if gain else None)
        line["sweep4"] = dict(sweep, frames=args.sweep_frames,
                              cells="scheduler+load: quad + infeasible frames")
        line["encoder"] = {"gflop_per_agent": sig(flops / 1e9), **{f"b{n}": [v["tflops"], v["frac"]]
                                                                  for n, v in enc_by_n.items()}}
        line["fusion"] = {"gbs": sig(fu_gbs), "frac": sig(fu_gbs / hbm, 3) if fu_gbs else None,
                          "mb": sig(fusion_bytes(cfg, K) / 1e6),
                          "us": sig(np.mean(fk_zero) * 1e3) if fk_zero else None,
                          "timing": "kernel's global-timer span, 8-agent frames"}
        line["pfn_us"] = sig(np.mean(pf) * 1e3) if pf else None
        line["release_ab_e2e"] = {k: {kk: vv[0] for kk, vv in v.items()} for k, v in ab.items()}
        line["multiscale_ms"] = msc
        line["gain_model"] = {"r": sig(gv["r"], 3), "mae_ms": sig(gv["mae_ms"], 3)}
        if args.detail:
            os.makedirs(os.path.dirname(os.path.abspath(args.detail)), exist_ok=True)
            with open(args.detail, "w") as f:
                json.dump({"line": line, "detail": detail}, f, default=_json_num, indent=1)
        print(json.dumps(line, default=_json_num, separators=(",", ":")), flush=True)
    if dist is not None:
        dist.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--sweep-frames", type=int, default=1000)
    ap.add_argument("--leg-frames", type=int, default=300)
    ap.add_argument("--detail", default=None)
    args = ap.parse_args()
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
