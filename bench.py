#!/usr/bin/env python
"""PRECOG hot-path benchmark on GB300.

One step = one pass of the whole hot path over one batch of synthetic input:
  * corpus encode of the paper-shaped workload: 24 independent layers (D=256,
    N=16), 4096 chunks x 3000 tokens, bf16 inputs, fp32 state, captured into a
    bf16 bank of 192 KB per chunk (C-ABI encode calls of S layers each, alternating
    over two streams so that each call's CTAs fill the previous call's last wave);
  * the query-time path: top-1 retrieval of a query batch over 1,000,000
    unit-norm fp16 keys of dim 768, injection of the retrieved 192 KB state from
    a 1,000,000-entry bank and scan prefill of 64 query tokens per query.

value = corpus tokens encoded per second (through all 24 layers) by all ranks.
The 24 layers' inputs (12.98 GB each, 311 GB in all) exceed HBM: `--input-sets`
S (default 4) independently generated layer inputs stay resident, contiguous,
and one encode call covers S layers, layer l reading set l mod S. Every layer
still streams its full 12.98 GB from HBM (far above the 129 MB L2), so the timed
traffic and work equal those of 24 independent layers; generating the synthetic
inputs is not part of the method and is timed separately. The retrieve+inject+prefill p50 latency is measured after the
timed steps, per query batch, with L2 flushed before every iteration (a 256 MB buffer written, then
a second one read, so the flush's dirty lines are written back outside the timed call); the same
calls replayed from a CUDA graph are reported beside it.

`--impl reference` times the CPU oracle (fp64, sequential) on a bounded sample
of the same workload on the host cores and prints the same JSON line.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "corpus-encode tokens/s & % HBM roofline; retrieve+inject+prefill p50 latency"
UNIT = "tokens/s"
FALLBACK_HBM_GBS = 6800.0
PROFILE = os.path.join(ROOT, "profiles", "scan_encode_paper_shaped.md")
SCAN_SRC = os.path.join(ROOT, "paper_2608_02560_gb300", "csrc", "scan.cu")


def parse_args():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--input-sets", type=int, default=4,
                    help="independent layer inputs kept resident; each encode call covers this many "
                         "layers (must divide 24)")
    ap.add_argument("--query-batch", type=int, default=1)
    ap.add_argument("--latency-iters", type=int, default=200)
    ap.add_argument("--e2e-steps", type=int, default=2)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--no-latency", action="store_true")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the single-layer wide and the ragged large-scale encode measurements")
    ap.add_argument("--no-extras", action="store_true",
                    help="skip the measurements of the extension rows (top-k, trajectory, complex A, SMC)")
    ap.add_argument("--case", choices=["full", "scan-small", "retrieve-small", "topk-small", "prefill-small",
                                       "wide-encode", "wide-encode-y", "ragged-encode", "trajectory-small",
                                       "complex-small", "consolidate"],
                    default="full",
                    help="small single-kernel cases (a few GB) used for profiler captures")
    return ap.parse_args()


def scan_bytes_per_launch(T, n_chunks, D, N, in_bytes=2, state_bytes=2):
    """Algorithmic HBM bytes of one encode launch: every input element read once
    (x, dt: T*D each; B: T*N), the captured state written once, the offsets and A read."""
    return T * (2 * D + N) * in_bytes + n_chunks * D * N * state_bytes + 8 * (n_chunks + 1) + 4 * D * N


def host_available_bytes() -> int:
    """MemAvailable of the host (0 if it cannot be read)."""
    try:
        with open("/proc/meminfo") as f:
            for line in f:
                if line.startswith("MemAvailable:"):
                    return int(line.split()[1]) * 1024
    except OSError:
        pass
    return 0


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        try:
            p = json.load(open(path))
            return float(p["hbm_gbs"]), "measured"
        except Exception:
            pass
    return FALLBACK_HBM_GBS, "fallback"


# FP32 lane operations one channel-token of the rescaled capture needs on the FMA pipe:
# the exponent sum L += dt * k (1), u = dt * x (1), the 16 weights u * E^(n+1) (16
# multiplies) and the 16 accumulations G_n += w_n * B_n (16 FMAs). The exponential E = 2^L
# runs on the SFU and is not counted.
ALU_OPS_PER_CHANNEL_TOKEN = 34
# The direct update with a readout (y mode): the exponent argument dt * A[d,0] (1), u = dt * x
# (1), the decay powers alpha_n = r^(n+1) (r^2 and 7 packed multiplies: 15), u * B_n (16),
# h_n = alpha_n h_n + u B_n (16 FMAs) and y = sum_n C_n h_n (16 FMAs and one add: 17).
ALU_OPS_DIRECT_Y = 66
FP32_LANES_PER_SM = 128      # 4 sub-partitions x 32 FP32 lanes (FFMA and FFMA2 alike)
FALLBACK_SM_MHZ = 2070.0


def alu_peak_tops(dev):
    """FP32 FMA-pipe peak in tera lane-operations per second: SMs x lanes x max SM clock."""
    import torch
    mhz = FALLBACK_SM_MHZ
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        try:
            mhz = float(json.load(open(path)).get("sm_max_mhz", mhz))
        except Exception:
            pass
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    return sms * FP32_LANES_PER_SM * mhz * 1e6 / 1e12, sms, mhz


def profiled_traffic():
    """DRAM traffic of one single-layer encode launch from the committed ncu summary, if
    it was taken on the current scan kernel source (else None)."""
    if not os.path.exists(PROFILE):
        return None
    text = open(PROFILE).read()
    m_sha = re.search(r"scan\.cu sha256:\s*([0-9a-f]{64})", text)
    m_tr = re.search(r"traffic_bytes_per_launch:\s*([0-9.eE+]+)", text)
    if not m_sha or not m_tr:
        return None
    sha = hashlib.sha256(open(SCAN_SRC, "rb").read()).hexdigest()
    return float(m_tr.group(1)) if sha == m_sha.group(1) else None


class Clocks:
    """Samples nvidia-smi clocks and throttle reasons while a region runs."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        rows = []
        if self.path and os.path.exists(self.path):
            for line in open(self.path):
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
            os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        power = [float(r[3]) for r in rows if re.match(r"^[0-9.]+$", r[3])]
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "power_w_max": max(power) if power else None, "samples": len(rows)}


# ------------------------------------------------------------------------------ ranks


def shard_seed(rank: int) -> int:
    """Seed of a rank's corpus shard. Chunks are encoded independently (Sec. 4.2), so every
    rank encodes its own chunks of the same shape: weak scaling, no exchange on the data
    path."""
    return 1000 * rank


def reduce_max(v: float, world: int, device) -> float:
    """The slowest rank's time (max over ranks); ``device`` is where the process group
    reduces (a CUDA device under NCCL, the CPU under gloo)."""
    if world == 1:
        return v
    import torch
    import torch.distributed as dist
    t = torch.tensor([v], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank_step: float, world: int, steps: int, seconds: float) -> float:
    """Units processed by all ranks per second of the slowest rank."""
    return world * units_per_rank_step * steps / seconds


# ------------------------------------------------------------------------------ reference arm


def run_reference(args):
    """The oracle (fp64; each chunk a sequential rollout, chunks split over every host
    core) on a bounded sample of the paper-shaped encode."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    import torch

    import oracle
    import synth
    shape = synth.PAPER
    cores = os.cpu_count() or 1
    chunks, T = 4 * cores, shape.chunk_len
    x, dt, A, B, _ = synth.host_scan_inputs(chunks * T, shape.D, shape.N, seed=0)
    # bf16 inputs, widened exactly, as the GPU path sees them
    bf = lambda a: torch.from_numpy(a).to(torch.bfloat16).double().numpy()
    x, dt, B = bf(x), bf(dt), bf(B)
    off = synth.fixed_offsets(chunks, T)
    oracle.build()
    for _ in range(args.warmup):
        oracle.scan_threads(x, dt, A, B, off, cores)
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        oracle.scan_threads(x, dt, A, B, off, cores)
        times.append(time.perf_counter() - t0)
    per_layer = chunks * T / statistics.mean(times)
    value = per_layer / shape.n_layers          # tokens through all 24 layers per second
    sample = (f"{chunks} chunks x {T} tokens x 1 layer of the paper-shaped encode (D=256, N=16) on "
              f"{cores} host threads, bf16-valued inputs in fp64; rate divided by 24 layers")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * statistics.mean(times), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": "paper-shaped corpus encode (sampled for the CPU oracle)",
                       "chunk_tokens": T, "layers": shape.n_layers, "D": shape.D, "N": shape.N},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------------------ profiler cases


def run_case(args):
    """Small cases of one kernel each, sized above L2 but a few GB on the device, for
    profiler captures: 3 launches of the kernel (the first is a warm-up)."""
    import torch

    import paper_2608_02560_gb300 as pg
    import synth
    dev = torch.device("cuda:0")
    res = {"case": args.case}
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(6)]
    if args.case == "scan-small":
        # paper-shaped rows (D=256, N=16, bf16) in 3040 chunks of 1000 tokens: 3.2 GB, about
        # 20 blocks per SM, so the per-token behaviour and occupancy match the full launch
        shape, chunks, clen = synth.PAPER, 3040, 1000
        off_np = synth.fixed_offsets(chunks, clen)
        T = int(off_np[-1])
        inp = synth.device_scan_inputs(T, shape.D, shape.N, 0, 0, dev, with_C=False)
        bank = torch.empty((chunks, shape.n_layers, shape.D, shape.N), dtype=torch.bfloat16, device=dev)
        off = torch.from_numpy(off_np).to(dev)
        si = pg.scan_inputs(inp["x"], inp["dt"], inp["B"], inp["A"], a_kind=pg.PRECOG_A_POWER)
        fn = lambda: pg.precog_encode_chunks(si, off, T, states_out=bank, layer0=0, L_total=shape.n_layers)
        res["algorithmic_bytes_per_launch"] = scan_bytes_per_launch(T, chunks, shape.D, shape.N)
        res["scale_to_full_launch"] = shape.n_chunks * shape.chunk_len / T
    elif args.case in ("trajectory-small", "complex-small"):
        # the scan-small rows (3040 chunks x 1000 tokens, D=256): every 250th state kept, or
        # the complex diagonal A of Eq. 1 (real part -(n+1), imaginary part pi*n)
        shape, chunks, clen = synth.PAPER, 3040, 1000
        off_np = synth.fixed_offsets(chunks, clen)
        T = int(off_np[-1])
        inp = synth.device_scan_inputs(T, shape.D, shape.N, 0, 0, dev, with_C=False)
        off = torch.from_numpy(off_np).to(dev)
        in_bytes = T * (2 * shape.D + shape.N) * 2
        if args.case == "trajectory-small":
            stride = 250
            eo = torch.arange(chunks + 1, dtype=torch.int64, device=dev) * (clen // stride)
            traj = torch.empty((chunks * (clen // stride), 1, shape.D, shape.N), dtype=torch.bfloat16, device=dev)
            si = pg.scan_inputs(inp["x"], inp["dt"], inp["B"], inp["A"], a_kind=pg.PRECOG_A_POWER)
            fn = lambda: pg.precog_encode_trajectory(si, off, T, stride, eo, traj)
            res["algorithmic_bytes_per_launch"] = in_bytes + traj.numel() * 2
        else:
            im = (math.pi * torch.arange(shape.N, device=dev, dtype=torch.float32)).expand(shape.D, shape.N)
            A = torch.complex(inp["A"], im).contiguous()
            cst = torch.empty((chunks, 1, shape.D, shape.N, 2), dtype=torch.bfloat16, device=dev)
            si = pg.scan_inputs(inp["x"], inp["dt"], inp["B"], A, a_kind=pg.PRECOG_A_COMPLEX)
            fn = lambda: pg.precog_encode_chunks(si, off, T, states_out=cst)
            res["algorithmic_bytes_per_launch"] = in_bytes + cst.numel() * 2
    elif args.case == "consolidate":
        # 4096 24-layer bf16 states (805 MB) folded into 64 semantic slots
        n, elems = 4096, 24 * 256 * 16
        states = synth.device_normal_bank(n, elems, 22, dev)
        slots = torch.arange(n, dtype=torch.int64, device=dev) * 7 % 64
        sem = torch.zeros((64, elems), dtype=torch.float32, device=dev)
        fn = lambda: pg.precog_smc_consolidate(sem, states, slots, 0.1)
        res["algorithmic_bytes_per_launch"] = n * elems * 2 + 2 * sem.numel() * 4
    elif args.case in ("wide-encode", "wide-encode-y", "ragged-encode"):
        # one layer of the single-layer wide encode (D=2048, 1024 x 512 tokens; capture or
        # readout) or of the ragged encode (D=512, 8192 chunks of 256..4096 tokens)
        shape = synth.RAGGED if args.case == "ragged-encode" else synth.WIDE
        y_mode = args.case == "wide-encode-y"
        off_np = synth.shape_offsets(shape, 0)
        T = int(off_np[-1])
        inp = synth.device_scan_inputs(T, shape.D, shape.N, 0, 0, dev, with_C=y_mode)
        off = torch.from_numpy(off_np).to(dev)
        sdt = torch.float32 if shape is synth.WIDE else torch.bfloat16
        bank = torch.empty((shape.n_chunks, 1, shape.D, shape.N), dtype=sdt, device=dev)
        y = torch.empty((1, T, shape.D), dtype=torch.bfloat16, device=dev) if y_mode else None
        si = pg.scan_inputs(inp["x"], inp["dt"], inp["B"], inp["A"], inp["C"] if y_mode else None,
                            a_kind=pg.PRECOG_A_POWER)
        fn = lambda: pg.precog_encode_chunks(si, off, T, states_out=bank, y_out=y)
        nb = scan_bytes_per_launch(T, shape.n_chunks, shape.D, shape.N, state_bytes=bank.element_size())
        if y_mode:
            nb += T * shape.N * 2 + T * shape.D * 2
        res["algorithmic_bytes_per_launch"] = nb
        res["tokens"] = T
    elif args.case in ("retrieve-small", "topk-small"):
        M = 1 << 18
        index = synth.device_unit_index(M, synth.QUERY_DIM, 0, dev)
        q, _ = synth.device_planted_queries(index, args.query_batch, synth.QUERY_NOISE, 1)
        if args.case == "retrieve-small":
            idx = torch.empty(args.query_batch, dtype=torch.int64, device=dev)
            fn = lambda: pg.precog_retrieve(index, q, idx)
        else:
            idx = torch.empty((args.query_batch, 3), dtype=torch.int64, device=dev)
            sc = torch.empty((args.query_batch, 3), dtype=torch.float32, device=dev)
            fn = lambda: pg.precog_retrieve_topk(index, q, 3, idx, sc)
        res["algorithmic_bytes_per_launch"] = M * synth.QUERY_DIM * 2
    else:
        L, D, N, Tq, Q, entries = 24, 256, 16, synth.QUERY_TOKENS, args.query_batch, 4096
        bank = synth.device_normal_bank(entries, L * D * N, 1, dev).view(entries, L, D, N)
        ins = [synth.device_scan_inputs(Q * Tq, D, N, 2, l, dev) for l in range(L)]
        st = lambda k: torch.stack([i[k] for i in ins]).contiguous()
        x, dt, B, C, A = st("x"), st("dt"), st("B"), st("C"), st("A")
        si = pg.scan_inputs(x, dt, B, A, C, a_kind=pg.PRECOG_A_POWER)
        idx = torch.arange(Q, dtype=torch.int64, device=dev) * 7 % entries
        y = torch.empty((L, Q * Tq, D), dtype=torch.bfloat16, device=dev)
        h = torch.empty((Q, L, D, N), dtype=torch.bfloat16, device=dev)
        fn = lambda: pg.precog_prefill_from_state(si, Q, Tq, bank, idx=idx, y_out=y, state_out=h)
    times = []
    for i in range(3):
        ev[2 * i].record()
        fn()
        ev[2 * i + 1].record()
    torch.cuda.synchronize()
    res["ms"] = [ev[2 * i].elapsed_time(ev[2 * i + 1]) for i in range(3)]
    if "algorithmic_bytes_per_launch" in res:
        best = min(res["ms"][1:])
        res["achieved_gbs"] = res["algorithmic_bytes_per_launch"] / (best * 1e-3) / 1e9
        res["frac_hbm"] = res["achieved_gbs"] / peaks()[0]
    st, bits = pg.precog_device_status()
    res["device_status"] = [st, bits]
    print(json.dumps(res), flush=True)
    if st != 0:
        sys.exit(1)


# ------------------------------------------------------------------------------ extension rows


def measure_extensions(pg, synth, torch, dev, layer_in, off, T, n_chunks, index, qbank, query_batch, hbm,
                       call_in=None, layers_per_call=1):
    """Times the extension rows on the resident paper-shaped buffers (a few seconds):
    top-k retrieval and composed prefill (Sec. 4.4), K-dial trajectory capture (Sec. 5.2),
    the complex-A scan (Eq. 1's complex diagonal) and the SMC routing / EMA kernels (Sec. 5).
    Each entry: median ms over a few launches (L2 flushed before each), algorithmic bytes
    (or flops) of one launch and the fraction of the measured peak they reach."""
    import numpy as np
    D, N = layer_in["x"].shape[1], layer_in["B"].shape[1]
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)

    evict = torch.empty_like(flush)

    def timed(fn, iters=5):
        fn()
        ts = []
        for _ in range(iters):
            flush.zero_()          # L2 flush; reading a second buffer writes its dirty lines back
            evict.sum()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            fn()
            b.record()
            b.synchronize()
            ts.append(a.elapsed_time(b))
        ts.sort()
        return ts[len(ts) // 2]

    def hbm_row(ms, nbytes, **kw):
        gbs = nbytes / (ms * 1e-3) / 1e9
        return dict(ms=ms, algorithmic_bytes=nbytes, achieved_gbs=gbs, frac_hbm=gbs / hbm, **kw)

    out = {}
    in_bytes = T * (2 * D + N) * 2
    # f2: trajectory, one state every 1000 tokens of each 3000-token chunk (K = 3)
    stride = 1000
    lens = (off[1:] - off[:-1]).cpu().numpy()
    eo_np = np.concatenate([[0], np.cumsum((lens + stride - 1) // stride)]).astype(np.int64)
    eo = torch.from_numpy(eo_np).to(dev)
    # as many layers per call as the encode (a launch's partial last wave is shared by them)
    S = layers_per_call if call_in is not None else 1
    traj = torch.empty((int(eo_np[-1]), S, D, N), dtype=torch.bfloat16, device=dev)
    si = call_in if call_in is not None else pg.scan_inputs(layer_in["x"], layer_in["dt"], layer_in["B"],
                                                            layer_in["A"], a_kind=pg.PRECOG_A_POWER)
    ms = timed(lambda: pg.precog_encode_trajectory(si, off, T, stride, eo, traj), 3)
    out["trajectory_stride1000"] = hbm_row(ms, S * in_bytes + traj.numel() * 2, entries=int(eo_np[-1]),
                                           layers_per_call=S, ms_per_layer=ms / S,
                                           tokens_per_s=S * T / (ms * 1e-3))
    del traj
    # a2 in its literal form: the same layer with A given as general (not stated as power
    # form), one SFU exponential per (token, channel, state index): 16 per channel-token at
    # 32 per clock per SM (measured) bound it
    sg = pg.scan_inputs(layer_in["x"], layer_in["dt"], layer_in["B"], layer_in["A"], a_kind=pg.PRECOG_A_GENERAL)
    gst = torch.empty((n_chunks, 1, D, N), dtype=torch.bfloat16, device=dev)
    ms = timed(lambda: pg.precog_encode_chunks(sg, off, T, states_out=gst), 3)
    props = torch.cuda.get_device_properties(dev)
    sfu_floor_ms = T * D * N / (props.multi_processor_count * 32 * 2.07e9) * 1e3
    out["encode_general_A"] = hbm_row(ms, in_bytes + gst.numel() * 2, tokens_per_s=T / (ms * 1e-3),
                                      bound="alu (SFU: one exponential per state update)",
                                      sfu_floor_ms_at_2070mhz=sfu_floor_ms, frac_sfu=sfu_floor_ms / ms)
    del gst
    # f3: complex A, paper parameterisation (real part -(n+1), imaginary part pi*n)
    A = torch.complex(layer_in["A"], (math.pi * torch.arange(N, device=dev, dtype=torch.float32)).expand(D, N))
    A = A.contiguous()
    sc = pg.scan_inputs(layer_in["x"], layer_in["dt"], layer_in["B"], A, a_kind=pg.PRECOG_A_COMPLEX)
    cst = torch.empty((n_chunks, 1, D, N, 2), dtype=torch.bfloat16, device=dev)
    ms = timed(lambda: pg.precog_encode_chunks(sc, off, T, states_out=cst), 3)
    # This A (real part -(n+1), imaginary part pi n in fp32) takes the power form, and a
    # capture without readout accumulates it rescaled: per state index one complex multiply
    # of the power tree of the weights (4 FP32 lane operations) and two real FMAs adding
    # w_n B_n to the rescaled state, i.e. 96 per channel-token on the FMA pipe (128 lane
    # operations per clock per SM); the per-token exponent, phase and scale are not counted.
    props = torch.cuda.get_device_properties(dev)
    alu_floor_ms = T * D * N * 6 / (props.multi_processor_count * 128 * 2.07e9) * 1e3
    out["complex_A_encode"] = hbm_row(ms, in_bytes + cst.numel() * 2, tokens_per_s=T / (ms * 1e-3),
                                      bound="alu (FMA pipe: rotation tree and complex update)",
                                      alu_floor_ms_at_2070mhz=alu_floor_ms, frac_alu=alu_floor_ms / ms)
    # Eq. 1's own parameterisation: real part -softplus(a) per state index (no power
    # structure), imaginary part pi*n: the harmonic form, accumulated rescaled in a capture:
    # per state index the rotation tree 4 FP32 lane operations on the FMA pipe, the
    # exponent's argument 1, the magnitude times B_n 1 and two FMAs into the rescaled state
    # 2, i.e. 8 (the exponential itself runs on the SFU)
    g = torch.Generator(device=dev)
    g.manual_seed(29)
    re = -torch.nn.functional.softplus(torch.randn((D, N), generator=g, device=dev))
    A = torch.complex(re, (math.pi * torch.arange(N, device=dev, dtype=torch.float32)).expand(D, N)).contiguous()
    sc = pg.scan_inputs(layer_in["x"], layer_in["dt"], layer_in["B"], A, a_kind=pg.PRECOG_A_COMPLEX)
    ms = timed(lambda: pg.precog_encode_chunks(sc, off, T, states_out=cst), 3)
    alu_floor_ms = T * D * N * 8 / (props.multi_processor_count * 128 * 2.07e9) * 1e3
    out["complex_A_encode_softplus_re"] = hbm_row(ms, in_bytes + cst.numel() * 2, tokens_per_s=T / (ms * 1e-3),
                                                  bound="alu (FMA pipe; one SFU exponential per state index)",
                                                  alu_floor_ms_at_2070mhz=alu_floor_ms, frac_alu=alu_floor_ms / ms)
    del cst
    # f1: top-3 retrieval over the 1M index and the composed 24-layer prefill
    M, dim = index.shape
    for nq in (1, 256):
        b = query_batch(nq, 4242 + nq)
        k = 3
        ti = torch.empty((nq, k), dtype=torch.int64, device=dev)
        ts_ = torch.empty((nq, k), dtype=torch.float32, device=dev)
        ws = torch.empty(pg.precog_retrieve_topk_workspace_size(M, dim, nq) + 16, dtype=torch.uint8, device=dev)
        ms_r = timed(lambda: pg.precog_retrieve_topk(index, b["q"], k, ti, ts_, workspace=ws))
        Tq = b["x"].shape[1] // nq
        ms_c = timed(lambda: pg.precog_prefill_composed(b["in"], nq, Tq, qbank, ti, ts_, k,
                                                        y_out=b["y"], state_out=b["h"]))
        row = hbm_row(ms_r, M * dim * 2, k=k, planted_first=bool(torch.equal(ti[:, 0], b["rows"])))
        if nq > 1:
            row["tflops"] = 2.0 * nq * M * dim / (ms_r * 1e-3) / 1e12
        out[f"topk_retrieve_q{nq}"] = row
        L = qbank.shape[1]
        cb = nq * k * L * D * N * 2 + b["x"].numel() * 4 + b["B"].numel() * 4 + b["y"].numel() * 2 + b["h"].numel() * 2
        out[f"composed_prefill_q{nq}_k3"] = hbm_row(ms_c, cb)
        del b, ws
    # f4: SMC routing of 4096 chunk embeddings into 16 domains x 64 sub-clusters, and the
    # EMA of 4096 captured 24-layer states into 64 semantic slots
    n_emb, Md, J = 4096, 16, 64
    emb = index[:n_emb]
    dom = index[n_emb:n_emb + Md].contiguous()
    sub = index[n_emb + Md:n_emb + Md + Md * J].contiguous().view(Md, J, dim)
    Jt = torch.full((Md,), J, dtype=torch.int32, device=dev)
    om = torch.empty(n_emb, dtype=torch.int32, device=dev)
    oj = torch.empty(n_emb, dtype=torch.int32, device=dev)
    os_ = torch.empty(n_emb, dtype=torch.int64, device=dev)
    ms = timed(lambda: pg.precog_smc_route(emb, dom, sub, Jt, om, oj, os_))
    out["smc_route_4096x(16+64)"] = dict(ms=ms, flops=2.0 * n_emb * (Md + J) * dim,
                                         l2_to_sm_bytes=n_emb * (Md + J) * dim * 2,
                                         note="each warp streams its embedding's 80 prototypes "
                                              "(120 KB) from L2, eight at a time")
    bank_states = qbank[:n_emb].view(n_emb, -1)
    sem = torch.zeros((J, bank_states.shape[1]), dtype=torch.float32, device=dev)
    slots = torch.arange(n_emb, dtype=torch.int64, device=dev) % J
    ms = timed(lambda: pg.precog_smc_consolidate(sem, bank_states, slots, 0.1), 3)
    out["smc_consolidate_4096_into_64"] = hbm_row(ms, bank_states.numel() * 2 + 2 * sem.numel() * 4)
    del sem, flush, evict
    return out


def measure_configs(pg, synth, torch, dev, hbm, alu_peak, cpu_chunks):
    """The two other encode workloads, each on its own resident inputs (every launch
    streams them from HBM; they are far above L2): the single-layer wide encode (D=2048,
    1024 x 512 tokens; fp32 state capture, and a readout mode writing bf16 y) and one layer
    of the ragged large-scale encode (D=512, 8192 chunks of U[256, 4096] tokens, bf16
    bank; 24 such layers make the workload). Returns the rows and, for the CPU baseline,
    the first ``cpu_chunks`` chunks of each workload's inputs copied back to the host."""
    import numpy as np
    out, samples = {}, {}

    def timed(fn, iters=5):
        fn()
        ts = []
        for _ in range(iters):
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            fn()
            b.record()
            b.synchronize()
            ts.append(a.elapsed_time(b))
        ts.sort()
        return ts[len(ts) // 2]

    for shape in (synth.WIDE, synth.RAGGED):
        off_np = synth.shape_offsets(shape, 0)
        T = int(off_np[-1])
        inp = synth.device_scan_inputs(T, shape.D, shape.N, 0, 0, dev, with_C=shape is synth.WIDE)
        off = torch.from_numpy(off_np).to(dev)
        sdt = torch.float32 if shape is synth.WIDE else torch.bfloat16
        states = torch.empty((shape.n_chunks, 1, shape.D, shape.N), dtype=sdt, device=dev)
        si = pg.scan_inputs(inp["x"], inp["dt"], inp["B"], inp["A"], a_kind=pg.PRECOG_A_POWER)
        if shape is synth.RAGGED:
            # ragged chunks are taken up longest first (the caller knows the lengths it laid
            # out), so the short ones fill the launch's tail; the unordered time is kept too
            order = torch.from_numpy(np.argsort(-np.diff(off_np), kind="stable").astype(np.int64)).to(dev)
            ms_unordered = timed(lambda: pg.precog_encode_chunks(si, off, T, states_out=states))
            ms = timed(lambda: pg.precog_encode_chunks_ordered(si, off, T, order, states_out=states))
        else:
            ms = timed(lambda: pg.precog_encode_chunks(si, off, T, states_out=states))
        nb = scan_bytes_per_launch(T, shape.n_chunks, shape.D, shape.N, state_bytes=states.element_size())
        ct = T * shape.D
        row = {"ms_per_layer": ms, "tokens": T, "chunks": shape.n_chunks, "D": shape.D,
               "algorithmic_bytes": nb, "achieved_gbs": nb / (ms * 1e-3) / 1e9,
               "frac_hbm": nb / (ms * 1e-3) / 1e9 / hbm,
               "frac_alu": ALU_OPS_PER_CHANNEL_TOKEN * ct / (ms * 1e-3) / 1e12 / alu_peak,
               "state_dtype": str(sdt).replace("torch.", "")}
        if shape is synth.WIDE:
            row["tokens_per_s"] = T / (ms * 1e-3)
            out["wide_encode_capture"] = row
            y = torch.empty((1, T, shape.D), dtype=torch.bfloat16, device=dev)
            sy = pg.scan_inputs(inp["x"], inp["dt"], inp["B"], inp["A"], inp["C"], a_kind=pg.PRECOG_A_POWER)
            ms = timed(lambda: pg.precog_encode_chunks(sy, off, T, states_out=states, y_out=y))
            nb_y = nb + T * shape.N * 2 + T * shape.D * 2
            out["wide_encode_y"] = {"ms_per_layer": ms, "tokens": T, "tokens_per_s": T / (ms * 1e-3),
                                    "algorithmic_bytes": nb_y, "achieved_gbs": nb_y / (ms * 1e-3) / 1e9,
                                    "frac_hbm": nb_y / (ms * 1e-3) / 1e9 / hbm,
                                    "frac_alu": ALU_OPS_DIRECT_Y * ct / (ms * 1e-3) / 1e12 / alu_peak,
                                    "alu_ops_per_channel_token": ALU_OPS_DIRECT_Y}
            del y
        else:
            row["layers"] = shape.n_layers
            row["tokens_per_s"] = T / (shape.n_layers * ms * 1e-3)   # through all 24 layers
            row["order"] = "longest chunk first (precog_encode_chunks_ordered)"
            row["ms_per_layer_unordered"] = ms_unordered
            out["ragged_encode"] = row
        r1 = int(off_np[cpu_chunks])
        samples[shape.name] = {k: inp[k][:r1].cpu().double().numpy() for k in ("x", "dt", "B")}
        samples[shape.name]["A"] = inp["A"].cpu().double().numpy()
        samples[shape.name]["offsets"] = off_np[:cpu_chunks + 1].copy()
        samples[shape.name]["per_layer_tokens"] = T
        samples[shape.name]["layers"] = shape.n_layers
        del inp, states, si
        torch.cuda.empty_cache()
    return out, samples


def cpu_baseline(oracle, paper, others, query, L):
    """The oracle (fp64, sequential per chunk) on bounded samples of each workload, on
    one host core and on every host core (chunks split over threads, each chunk the same
    sequential rollout). Rates are extrapolated linearly: chunks and layers are
    independent (Sec. 4.2)."""
    oracle.build()
    cores = os.cpu_count() or 1

    def rate(sample, threads, chunks):
        off = sample["offsets"][:chunks + 1]
        r1 = int(off[-1])
        args = (sample["x"][:r1], sample["dt"][:r1], sample["A"], sample["B"][:r1], off)
        t0 = time.perf_counter()
        if threads == 1:
            oracle.scan(*args)
        else:
            oracle.scan_threads(*args, threads)
        dt_s = time.perf_counter() - t0
        return r1 / dt_s / sample["layers"], dt_s, r1

    res = {"kind": "oracle", "unit": UNIT, "cores": cores}
    one, s1, tok1 = rate(paper, 1, 16)
    n_all = paper["offsets"].shape[0] - 1
    allc, sa, toka = rate(paper, cores, n_all)
    res.update(value=allc, seconds=sa,
               sample=f"{n_all} chunks x 3000 tokens x 1 layer of the paper-shaped encode on {cores} host "
                      f"threads (chunks split across threads, fp64 sequential rollout per chunk); rate "
                      f"divided by {L} layers",
               single_core={"value": one, "seconds": s1, "sample": "16 chunks x 3000 tokens x 1 layer, one core"})
    for name, smp in others.items():
        n = smp["offsets"].shape[0] - 1
        o1, t1, _ = rate(smp, 1, min(n, 16))
        oa, ta, _ = rate(smp, cores, n)
        res[name] = {"single_core": o1, "all_cores": oa, "seconds": [t1, ta],
                     "sample": f"{min(n, 16)} chunks x 1 layer on one core, {n} chunks x 1 layer on "
                               f"{cores} threads; rates divided by {smp['layers']} layer(s)"}
    if query is not None:
        t0 = time.perf_counter()
        idx, _ = oracle.retrieve(query["index"], query["q"])
        t_r = time.perf_counter() - t0
        row = int(idx[0])
        t0 = time.perf_counter()
        for l in range(L):
            oracle.rollout(query["x"][l], query["dt"][l], query["A"][l], query["B"][l], query["C"][l],
                           h0=query["bank"][l], want_y=True)
        t_p = time.perf_counter() - t0
        res["query_path_q1"] = {"retrieve_s": t_r, "prefill_s": t_p, "latency_us": 1e6 * (t_r + t_p),
                                "retrieved_planted": row == query["row"],
                                "sample": "one query: exact retrieval over the full 1M x 768 index and "
                                          f"the {L}-layer prefill of 64 tokens from the injected state, "
                                          "one core"}
    return res


# ------------------------------------------------------------------------------ our arm


def main():
    args = parse_args()
    if args.impl == "reference":
        run_reference(args)
        return
    if args.case != "full":
        run_case(args)
        return
    import torch

    import paper_2608_02560_gb300 as pg
    import synth

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    pg.load_library()

    def barrier():
        if world > 1:
            torch.distributed.barrier()

    def max_over_ranks(v):
        return reduce_max(v, world, dev)

    shape = synth.PAPER
    L, D, N = shape.n_layers, shape.D, shape.N
    seed = shard_seed(rank)
    off_np = synth.shape_offsets(shape, seed)
    T = int(off_np[-1])
    off = torch.from_numpy(off_np).to(dev)

    # S independently drawn layer inputs, contiguous so that one C-ABI call encodes S
    # layers (S x 4096 CTAs: fewer partial last waves than one layer per launch)
    S = args.input_sets
    if S < 1 or L % S:
        raise SystemExit(f"--input-sets must divide {L}")
    t_gen = time.perf_counter()
    x_all = torch.empty((S, T, D), dtype=torch.bfloat16, device=dev)
    dt_all = torch.empty_like(x_all)
    B_all = torch.empty((S, T, N), dtype=torch.bfloat16, device=dev)
    sets = [synth.device_scan_inputs(T, D, N, seed, s, dev, with_C=False,
                                     out={"x": x_all[s], "dt": dt_all[s], "B": B_all[s]})
            for s in range(S)]
    torch.cuda.synchronize()
    gen_s_per_layer = (time.perf_counter() - t_gen) / S
    bank = torch.empty((shape.n_chunks, L, D, N), dtype=torch.bfloat16, device=dev)
    A_all = torch.stack([st["A"] for st in sets]).contiguous()
    call_in = pg.scan_inputs(x_all, dt_all, B_all, A_all, a_kind=pg.PRECOG_A_POWER)
    scan_in = [pg.scan_inputs(st["x"], st["dt"], st["B"], st["A"], a_kind=pg.PRECOG_A_POWER) for st in sets]
    calls = L // S

    # query-time workload. One rank: the whole index and bank. Several ranks: the index
    # and the bank are sharded by rows (each rank holds M / world of each); every rank
    # serves the same queries, retrieving over its rows, combining the shards' keys with
    # one all-reduce MAX and receiving the winning states from their owners (an all-reduce
    # of owner-filled rows) before it prefills.
    M, dim, Tq, Q = synth.QUERY_INDEX_M, synth.QUERY_DIM, synth.QUERY_TOKENS, args.query_batch
    qseed0 = 1 if world > 1 else seed          # the same index and queries on every rank
    index_full = synth.device_unit_index(M, dim, qseed0 + 1, dev)
    if world > 1:
        from paper_2608_02560_gb300 import distributed as pgd
        row_off, rows_here = pgd.shard_rows(M, world, rank)
        index = index_full[row_off:row_off + rows_here].clone()
        qbank = synth.device_normal_bank(rows_here, L * D * N, 2 + 1000 * rank, dev).view(rows_here, L, D, N)
    else:
        row_off, rows_here = 0, M
        index = index_full
        qbank = synth.device_normal_bank(M, L * D * N, seed + 2, dev).view(M, L, D, N)

    def query_batch(nq, qseed):
        q, rows = synth.device_planted_queries(index_full, nq, synth.QUERY_NOISE, qseed)
        ins = [synth.device_scan_inputs(nq * Tq, D, N, qseed, l, dev) for l in range(L)]
        st = lambda k: torch.stack([i[k] for i in ins]).contiguous()
        qx, qdt, qB, qC, qA = st("x"), st("dt"), st("B"), st("C"), st("A")
        out = {"q": q, "rows": rows, "x": qx, "dt": qdt, "B": qB, "C": qC, "A": qA,
               "in": pg.scan_inputs(qx, qdt, qB, qA, qC, a_kind=pg.PRECOG_A_POWER),
               "idx": torch.empty(nq, dtype=torch.int64, device=dev),
               "score": torch.empty(nq, dtype=torch.float32, device=dev),
               "ws": torch.empty(pg.precog_retrieve_workspace_size(rows_here, dim, nq) + 16,
                                 dtype=torch.uint8, device=dev),
               "inj": torch.empty((nq, L, D, N), dtype=torch.bfloat16, device=dev) if world > 1 else None,
               "y": torch.empty((L, nq * Tq, D), dtype=torch.bfloat16, device=dev),
               "h": torch.empty((nq, L, D, N), dtype=torch.bfloat16, device=dev), "n": nq}
        return out

    qb = query_batch(Q, qseed0 + 3)

    def query_path(b, stream=None):
        if world > 1:
            # torch's current stream carries the kernels and the collectives
            pgd.sharded_retrieve(index, b["q"], row_off, b["idx"], b["score"], workspace=b["ws"])
            pgd.gather_owned_states(qbank, row_off, b["idx"], b["inj"])
            pg.precog_prefill_from_state(b["in"], b["n"], Tq, b["inj"], idx=None, y_out=b["y"],
                                         state_out=b["h"])
            return
        pg.precog_retrieve(index, b["q"], b["idx"], b["score"], workspace=b["ws"], stream=stream)
        pg.precog_prefill_from_state(b["in"], b["n"], Tq, qbank, idx=b["idx"], y_out=b["y"],
                                     state_out=b["h"], stream=stream)

    # encode span of every timed step: from before its first encode launch to after both
    # streams' last one, on the main stream
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    side = torch.cuda.Stream(device=dev)
    fork, join = torch.cuda.Event(), torch.cuda.Event()

    def step(k=None):
        # layers c*S .. c*S+S-1 in one call; layer l reads input set l mod S. The calls write
        # disjoint layers of the bank and only read the input sets, so they alternate over
        # two streams: each call's CTAs take the SM slots that the previous call's last wave
        # frees, instead of waiting for all of it.
        main = torch.cuda.current_stream(dev)
        if k is not None:
            ev[k][0].record(main)
        fork.record(main)
        side.wait_event(fork)
        for c in range(calls):
            pg.precog_encode_chunks(call_in, off, T, states_out=bank, layer0=c * S, L_total=L,
                                    stream=main if c % 2 == 0 else side)
        join.record(side)
        main.wait_event(join)
        if k is not None:
            ev[k][1].record(main)
        query_path(qb)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    st, bits = pg.precog_device_status()
    if st != 0:
        raise RuntimeError(f"device status {st} bits {bits:#x} after warm-up")
    ok_rows = bool(torch.equal(qb["idx"], qb["rows"]))

    # ---------------- timed region
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    launches0 = pg.load_library().precog_launch_count()
    with Clocks(local_rank) as clk:
        barrier()
        torch.cuda.synchronize()
        t0.record()
        for k in range(args.steps):
            step(k)
        t1.record()
        torch.cuda.synchronize()
        barrier()
    launches = pg.load_library().precog_launch_count() - launches0
    clocks = clk.summary()
    elapsed_ms = max_over_ranks(t0.elapsed_time(t1))
    # per launch: the encode span of a step over its launches (the launches overlap by a wave)
    scan_ms = [a.elapsed_time(b) / calls for a, b in ev]
    tokens_per_step = T
    value = whole_job_rate(tokens_per_step, world, args.steps, elapsed_ms * 1e-3)
    ms_per_step = elapsed_ms / args.steps

    hbm, peak_src = peaks()
    bpl = S * scan_bytes_per_launch(T, shape.n_chunks, D, N)
    avg_scan_ms = statistics.mean(scan_ms)
    achieved = bpl / (avg_scan_ms * 1e-3) / 1e9
    layer_traffic = profiled_traffic()
    # The metric's roofline: algorithmic HBM bytes per launch over the launch's CUDA-event
    # time, against the measured copy bandwidth. The kernel's binding resource is the FP32
    # FMA pipe (ncu: FMA pipe busy, DRAM far from saturated), so the FMA-pipe roofline is
    # carried beside it, with the HBM fraction that pipe allows at 100 % busy.
    alu_peak, sms, mhz = alu_peak_tops(dev)
    ops = S * T * D * ALU_OPS_PER_CHANNEL_TOKEN
    alu_achieved = ops / (avg_scan_ms * 1e-3) / 1e12
    roofline = {"bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s", "frac": achieved / hbm,
                "peak_source": peak_src,
                "traffic": None if layer_traffic is None else S * layer_traffic,
                "traffic_source": ("dram__bytes_read.sum + dram__bytes_write.sum of the ncu capture "
                                   "summarised in profiles/scan_encode_paper_shaped.md (taken on this "
                                   "scan.cu, scaled by tokens to one launch)") if layer_traffic is not None
                else "null: the committed ncu capture was taken on another scan.cu",
                "limiter": "alu",
                "alu": {"achieved": alu_achieved, "peak": alu_peak,
                        "unit": "Tops/s (FP32 FMA-pipe lane operations)", "frac": alu_achieved / alu_peak,
                        "peak_derivation": f"{sms} SMs x {FP32_LANES_PER_SM} FP32 lanes x {mhz:.0f} MHz",
                        "ops_per_channel_token": ALU_OPS_PER_CHANNEL_TOKEN,
                        "algorithmic_ops_per_launch": ops,
                        "hbm_frac_at_alu_peak": alu_peak * 1e12 / ALU_OPS_PER_CHANNEL_TOKEN
                        * (bpl / (S * T * D)) / (hbm * 1e9)},
                "layers_per_launch": S,
                "kernel": "scan_kernel (encode, rescaled capture)",
                "algorithmic_bytes_per_launch": bpl, "avg_launch_ms": avg_scan_ms,
                "avg_launch_ms_source": (f"CUDA events around the {calls} encode launches of each timed step "
                                         "(alternating over two streams, joined) / launches")}

    # ---------------- end to end: host inputs -> device -> encode/query -> host results
    # (measured right after the timed steps: it is bound by the host link, and the later
    # latency and extension phases are not part of it)
    e2e = None
    if not args.no_e2e:
        # one pinned host copy per resident input set, so that layer l streams set l mod S's
        # inputs from the host and the e2e bank equals the timed region's
        # (when the host cannot pin that much for every rank on it, the sets share one copy)
        set_bytes = sum(sets[0][k].numel() * sets[0][k].element_size() for k in ("x", "dt", "B"))
        local_ranks = int(os.environ.get("LOCAL_WORLD_SIZE", "1"))
        HS = S if host_available_bytes() > 2 * S * set_bytes * local_ranks else 1
        host = [{k: torch.empty(sets[s_][k].shape, dtype=sets[s_][k].dtype, pin_memory=True)
                 for k in ("x", "dt", "B")} for s_ in range(HS)]
        for s_ in range(HS):
            for k in host[s_]:
                host[s_][k].copy_(sets[s_][k])
        host = [host[s_ % HS] for s_ in range(S)]
        hq = {k: torch.empty(qb[k].shape, dtype=qb[k].dtype, pin_memory=True)
              for k in ("q", "x", "dt", "B", "C")}
        for k in hq:
            hq[k].copy_(qb[k])
        bank_host = torch.empty(bank.shape, dtype=bank.dtype, pin_memory=True)
        out_host = {k: torch.empty(qb[k].shape, dtype=qb[k].dtype, pin_memory=True)
                    for k in ("idx", "score", "y", "h")}
        copy_stream = torch.cuda.Stream(device=dev)
        comp = torch.cuda.current_stream(dev)
        h2d = sum(host[l % S][k].numel() * host[l % S][k].element_size() for l in range(L) for k in host[0])
        h2d += sum(hq[k].numel() * hq[k].element_size() for k in hq)
        d2h = bank.numel() * bank.element_size()
        d2h += sum(out_host[k].numel() * out_host[k].element_size() for k in out_host)

        def e2e_step():
            done = [None] * S              # encode of the layer that last used each buffer
            copied = []
            for l in range(L):
                buf = sets[l % S]
                with torch.cuda.stream(copy_stream):
                    if done[l % S] is not None:
                        copy_stream.wait_event(done[l % S])
                    for k in ("x", "dt", "B"):
                        buf[k].copy_(host[l % S][k], non_blocking=True)
                    e = torch.cuda.Event()
                    e.record(copy_stream)
                comp.wait_event(e)
                pg.precog_encode_chunks(scan_in[l % S], off, T, states_out=bank, layer0=l, L_total=L)
                d = torch.cuda.Event()
                d.record(comp)
                done[l % S] = d
            for k in ("q", "x", "dt", "B", "C"):
                qb[k].copy_(hq[k], non_blocking=True)
            query_path(qb)
            bank_host.copy_(bank, non_blocking=True)
            for k in out_host:
                out_host[k].copy_(qb[k], non_blocking=True)

        e2e_step()
        torch.cuda.synchronize()
        barrier()
        w0 = time.perf_counter()
        for _ in range(args.e2e_steps):
            e2e_step()
        torch.cuda.synchronize()
        e2e_s = max_over_ranks(time.perf_counter() - w0)
        barrier()
        bank_matches = bool(torch.equal(bank_host, bank.cpu()))
        e2e = {"value": whole_job_rate(tokens_per_step, world, args.e2e_steps, e2e_s), "unit": UNIT,
               "host_input_sets": HS, "bank_equals_timed_region": bank_matches,
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
               "ms_per_step": 1e3 * e2e_s / args.e2e_steps, "steps": args.e2e_steps,
               # the host link is shared with the machine's other GPUs: this rate (and so
               # the e2e value) varies between runs
               "h2d_achieved_gbs": h2d * args.e2e_steps / e2e_s / 1e9}
        del host, hq, bank_host, out_host

    # ---------------- query latency (retrieve + inject + prefill), L2 flushed before each
    # call: a 256 MB buffer is written, then a second one read, so that the flush's dirty
    # lines are written back before the timed call instead of during it. The calls are
    # made eagerly through the API; the same calls captured in a CUDA graph are timed too.
    latency = {}
    if not args.no_latency:
        flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
        evict = torch.empty(256 << 20, dtype=torch.uint8, device=dev)

        def cold_l2():
            flush.zero_()
            evict.sum()

        def p50_p90(run, iters):
            times = []
            for _ in range(iters):
                cold_l2()
                s_ev, e_ev = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                s_ev.record()
                run()
                e_ev.record()
                e_ev.synchronize()
                times.append(s_ev.elapsed_time(e_ev) * 1e3)
            times.sort()
            return times[len(times) // 2], times[int(len(times) * 0.9)]

        for nq, iters in ((1, args.latency_iters), (256, max(20, args.latency_iters // 4))):
            b = qb if nq == Q else query_batch(nq, qseed0 + 7 + nq)
            for _ in range(3):
                query_path(b)
            p50, p90 = p50_p90(lambda: query_path(b), iters)
            g50 = None
            if world == 1:
                side = torch.cuda.Stream()
                side.wait_stream(torch.cuda.current_stream())
                with torch.cuda.stream(side):
                    query_path(b)
                torch.cuda.current_stream().wait_stream(side)
                graph = torch.cuda.CUDAGraph()
                with torch.cuda.graph(graph):
                    query_path(b)
                g50, _ = p50_p90(graph.replay, iters)
                del graph
            # the index sweep alone, at the measured copy bandwidth, bounds the latency below
            floor_us = rows_here * dim * index.element_size() / (peaks()[0] * 1e9) * 1e6
            latency[f"q{nq}"] = {"p50_us": p50, "p90_us": p90, "iters": iters,
                                 "graph_p50_us": g50, "index_sweep_floor_us": floor_us,
                                 "retrieved_planted": bool(torch.equal(b["idx"], b["rows"]))}
            if world > 1:
                latency[f"q{nq}"]["index_rows_per_rank"] = rows_here
            if b is not qb:
                del b
        del flush, evict

    # the extension rows and the other configurations are single-GPU measurements
    extras = None
    if not args.no_extras and world == 1:
        extras = measure_extensions(pg, synth, torch, dev, sets[0], off, T, shape.n_chunks, index, qbank,
                                    query_batch, peaks()[0], call_in=call_in, layers_per_call=S)

    st, bits = pg.precog_device_status()
    if st != 0:
        raise RuntimeError(f"device status {st} bits {bits:#x} after the timed region")

    # ---------------- CPU samples: the device-generated inputs of a few chunks (and of one
    # query) copied back, so the oracle sees exactly the values the GPU saw
    want_cpu = not args.no_cpu and rank == 0 and world == 1
    cpu_paper = cpu_query = None
    n_cpu = 16
    if want_cpu:
        n_paper = max(n_cpu, 16 * (os.cpu_count() or 1))
        r1 = n_paper * shape.chunk_len
        cpu_paper = {k: sets[0][k][:r1].cpu().double().numpy() for k in ("x", "dt", "B")}
        cpu_paper.update(A=sets[0]["A"].cpu().double().numpy(), offsets=synth.fixed_offsets(n_paper, shape.chunk_len),
                         layers=L)
        q1 = query_batch(1, seed + 11)
        prow = int(q1["rows"][0])
        cpu_query = {"index": index.cpu().double().numpy(), "q": q1["q"].cpu().double().numpy(),
                     "row": prow, "bank": qbank[prow].cpu().double().numpy(),
                     **{k: q1[k].cpu().double().numpy() for k in ("x", "dt", "B", "C", "A")}}
        del q1

    # ---------------- the other encode configurations, on their own resident inputs
    configs = None
    if not args.no_configs and world == 1:
        del x_all, dt_all, B_all, sets, call_in, scan_in, qbank, index, index_full, bank, qb
        torch.cuda.empty_cache()
        alu_peak_v = alu_peak_tops(dev)[0]
        configs, cfg_samples = measure_configs(pg, synth, torch, dev, peaks()[0], alu_peak_v,
                                               max(n_cpu, 4 * (os.cpu_count() or 1)))
        st, bits = pg.precog_device_status()
        if st != 0:
            raise RuntimeError(f"device status {st} bits {bits:#x} after the configuration runs")
    else:
        cfg_samples = {}

    # ---------------- CPU baseline: the oracle on bounded samples (rank 0, N=1 only)
    cpu = None
    if want_cpu:
        import oracle
        cpu = cpu_baseline(oracle, cpu_paper, cfg_samples, cpu_query, L)

    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
                "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
                "dtype": "f32", "io_dtype": "bf16", "data": "synthetic",
                "config": {"workload": "paper-shaped corpus encode + query-time path",
                           "layers": L, "D": D, "N": N, "chunks": shape.n_chunks,
                           "chunk_tokens": shape.chunk_len, "state_bytes_per_chunk": L * D * N * 2,
                           "input_sets_resident": S, "layers_per_encode_call": S,
                           "index_rows": M, "index_dim": dim, "bank_entries": M,
                           "query_batch": Q, "query_tokens": Tq, "parallelism": f"dp{world}",
                           "query_path": ("index and bank rows sharded over the ranks; one all-reduce MAX of "
                                          "the shards' keys, the winning states gathered by an all-reduce of "
                                          "owner-filled rows") if world > 1 else "whole index and bank on one GPU",
                           "l2": "inputs larger than L2 (12.98 GB per layer, 1.5 GB index)"},
                "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "clocks": clocks,
                "gpu_launches": int(launches), "latency": latency,
                "retrieved_planted": ok_rows, "input_gen_s_per_layer": gen_s_per_layer,
                "configs": configs, "extensions": extras}
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
