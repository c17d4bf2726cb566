#!/usr/bin/env python
"""Throughput of the Q-CNN test-phase forward on GB300.

Workload: AlexNet-shaped (ungrouped, CaffeNet-style) Q-CNN, batch 128 per GPU:
conv1 11x11/4 (C's=3, K=128), conv2 5x5 p2, conv3-5 3x3 p1 (C's=4, K=128),
3x3/2 max-pools, fc6-8 (C's=4, K=32); seeded synthetic images and
random-initialised codebooks/codes/biases (synth.alexnet()).  A step is one
forward of one batch through qcnn_net_forward (every layer, every stage).

Prints ONE JSON line (rank 0).  `--impl reference` times the float64 CPU
oracle on the same workload instead (the reference arm).
"""
from __future__ import annotations

import argparse
import json
import math
import multiprocessing as mp
import os
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import synth  # noqa: E402

METRIC = ("Q-CNN layer/net images/sec and dense-equiv GFLOP/s at batch 1/128; "
          "% of per-stage roofline")
WORKLOAD = "alexnet_qcnn"
BATCH = 128


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=30)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", choices=["qcnn", "reference"], default="qcnn")
    p.add_argument("--batch", type=int, default=BATCH)
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-extras", action="store_true",
                   help="skip the model-blob and quantizer measurements")
    p.add_argument("--cpu-sample", type=int, default=0,
                   help="images in the CPU-baseline sample (default: one per worker)")
    p.add_argument("--layer", default="",
                   help="WORKLOAD:INDEX -- time that one layer alone at --batch (warm-up, "
                        "then --steps launches; for profiling) and print one JSON line")
    return p.parse_args()


# ----------------------------------------------------------------- oracle
_CACHE = {}


def _workload_cache(batch):
    """Per-process copy of the workload's parameters and input batch."""
    if _CACHE.get("batch") != batch:
        w = synth.WORKLOADS[WORKLOAD]
        params = w.params()
        _CACHE.update(batch=batch, x=w.input(batch),
                      layers=[synth.oracle_layer_dict(L, P) for L, P in zip(w.layers, params)])
    return _CACHE


def _oracle_worker(args):
    """Run the float64 oracle on image `i` of the workload (spawned process)."""
    i, batch = args
    sys.path.insert(0, ROOT)
    import oracle as orc
    c = _workload_cache(batch)
    t = time.perf_counter()
    orc.net_forward(c["x"][i:i + 1], c["layers"])
    return time.perf_counter() - t


def _oracle_job(args):
    """Time the float64 oracle on n seeded images of workload `name` (spawned
    process; the images are drawn per job, so no batch is held)."""
    name, salt, n = args
    sys.path.insert(0, ROOT)
    import oracle as orc
    w = synth.WORKLOADS[name]
    key = ("layers", name)
    if key not in _CACHE:
        _CACHE[key] = [synth.oracle_layer_dict(L, P) for L, P in zip(w.layers, w.params())]
    x = w.input(n, 1000 + salt)
    t = time.perf_counter()
    orc.net_forward(x, _CACHE[key])
    return time.perf_counter() - t


def oracle_configs(pool, cores):
    """The oracle beside every workload: one image (the smallest batch of the
    workload when it is above 1) on one core, alone; and for workloads with
    a large batch, images spread over all `cores` processes (images/s)."""
    out = {}
    for name in sorted(synth.WORKLOADS):
        w = synth.WORKLOADS[name]
        b0 = min(w.batches)
        t1 = pool.apply(_oracle_job, ((name, 0, b0),))
        r = {"single_thread": {"batch": b0, "s": round(t1, 4),
                               "images_per_s": round(b0 / t1, 3)}}
        big = max(w.batches)
        if big > 8:
            sample = cores * (4 if t1 < 0.5 else 1)
            t = time.perf_counter()
            pool.map(_oracle_job, [(name, i + 1, 1) for i in range(sample)], chunksize=1)
            dt = time.perf_counter() - t
            r["all_cores"] = {"batch": big, "images": sample, "cores": cores,
                              "wall_s": round(dt, 3), "images_per_s": round(sample / dt, 3)}
        out[name] = r
    return out


def _cpu_info():
    model = ""
    try:
        for line in open("/proc/cpuinfo"):
            if line.lower().startswith(("model name", "cpu part", "hardware")):
                model = line.split(":", 1)[1].strip()
                break
    except OSError:
        pass
    return model


def oracle_pool(cores, batch):
    import oracle as orc
    orc.build()
    ctx = mp.get_context("spawn")
    pool = ctx.Pool(cores)
    pool.map(_oracle_ping, [batch] * cores, chunksize=1)
    return pool


def _oracle_ping(batch):
    sys.path.insert(0, ROOT)
    import oracle as orc
    orc.default()
    _workload_cache(batch)
    time.sleep(0.5)  # keep every worker busy so each one gets a ping
    return 0


def time_oracle(pool, cores, sample, batch):
    """Wall time of `sample` images through the oracle on `cores` processes."""
    t = time.perf_counter()
    pool.map(_oracle_worker, [(i % batch, batch) for i in range(sample)], chunksize=1)
    return time.perf_counter() - t


def reference_arm(a):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    cores = min(os.cpu_count() or 1, 16)
    pool = oracle_pool(cores, a.batch)
    sample = cores
    for _ in range(a.warmup):
        time_oracle(pool, cores, sample, a.batch)
    tot = 0.0
    for _ in range(a.steps):
        tot += time_oracle(pool, cores, sample, a.batch)
    pool.close()
    value = sample * a.steps / tot
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "images/s",
        "n_gpus": a.gpus, "steps": a.steps, "warmup": a.warmup,
        "ms_per_step": 1e3 * tot / a.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": WORKLOAD, "global_batch": a.batch, "images_per_step": sample},
        "cpu_baseline": {"value": value, "unit": "images/s", "cores": cores, "kind": "oracle",
                         "sample": f"{sample} images of the batch-{a.batch} workload per step, "
                                   f"one image per process, {cores} spawned processes, "
                                   f"float64 C oracle, host {_cpu_info()}"},
        "e2e": {"value": value, "unit": "images/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ------------------------------------------------------------------ clocks
class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
            time.sleep(0.6)
        except OSError:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.perf_counter(), line.strip()))

    def mark(self):
        return time.perf_counter()

    def stop(self, t0, t1):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.15)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = []
        for t, line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) != 7:
                continue
            try:
                rows.append((t, float(parts[0]), float(parts[1]), parts[3:]))
            except ValueError:
                continue
        inside = [r for r in rows if t0 - 0.06 <= r[0] <= t1 + 0.06] or rows
        if not inside:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in inside for i, v in enumerate(r[3]) if v.lower() == "active"})
        return {"sm_mhz": float(np.median([r[1] for r in inside])),
                "sm_max_mhz": max(r[2] for r in inside), "reasons": reasons,
                "samples": len(inside)}


# -------------------------------------------------------------- our arm
def load_peaks():
    try:
        return json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except (OSError, ValueError):
        return {}


def max_over_ranks(x: float, device) -> float:
    """The largest value of x over all ranks (the slowest rank's time)."""
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(images_per_rank: int, world: int, steps: int, seconds: float) -> float:
    """Whole-job images/s: every rank processes its own batch each step
    (independent replicas, weak scaling), timed by the slowest rank."""
    return images_per_rank * world * steps / seconds


def recorded_traffic(workload, batch, layer):
    """DRAM bytes per launch of a layer's kernel from the ncu record in
    profiles/dram_traffic.txt, or None when there is no record or the
    kernel's sources changed since it was taken."""
    import hashlib
    try:
        lines = open(os.path.join(ROOT, "profiles", "dram_traffic.txt")).read().splitlines()
    except OSError:
        return None
    for line in lines:
        if not line.strip() or line.startswith("#"):
            continue
        r = json.loads(line)
        if (r["workload"], r["batch"], r["layer"]) != (workload, batch, layer):
            continue
        h = hashlib.sha256()
        for s in r["sources"]:
            h.update(open(os.path.join(ROOT, s), "rb").read())
        if h.hexdigest() == r["sha256"]:
            return r["dram_read_bytes"] + r["dram_write_bytes"]
    return None


def extra_measurements(a, q, torch, w, params, x, out, flush, stream, dev, N, batch1, cm,
                       with_oracle):
    """The rows beyond the forward path: the stack loaded from a model blob
    (codes in ceil(log2 K) bits), and the quantizers (k-means, Eq. 4/6;
    error correction, Eq. 8-12), each timed on the GPU and, on rank 0 of a
    single-GPU run, the float64 oracle on one layer beside it."""
    import numpy as np

    res = {}

    def event_ms(fn, reps, flush_each=True):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        ts = []
        for _ in range(reps):
            if flush_each:
                flush.zero_()
            e0.record(stream)
            fn()
            e1.record(stream)
            torch.cuda.synchronize(dev)
            ts.append(e0.elapsed_time(e1))
        return float(np.median(ts))

    # ---- model blob
    layers = [synth.oracle_layer_dict(L, P) for L, P in zip(w.layers, params)]
    blob = q.serialize_model(layers, w.in_shape)
    lnet = q.load_model(blob, dev)
    lws = lnet.alloc_workspace(N, dev)
    for _ in range(3):
        lnet.forward(x, out=out, workspace=lws)
    torch.cuda.synchronize(dev)
    steps = max(5, a.steps // 3)
    ms = event_ms(lambda: lnet.forward(x, out=out, workspace=lws), steps)
    dense = sum(c.dense_bytes for c in _layer_costs(w, cm))
    res["model_blob"] = {
        "bytes": len(blob), "dense_fp32_weight_bytes": int(dense),
        "compression": round(dense / len(blob), 2),
        "note": "codes in ceil(log2 K) bits (Table 1 storage), sub-codebooks and biases fp32; "
                "FC layers of the loaded stack read the bit-packed codes directly",
        "value": round(N / (ms / 1e3), 1), "unit": "images/s", "ms_per_step": round(ms, 4),
        "batch1": batch1(lnet)}
    # fc6 at batch 1, byte codes vs packed rows (L2 flushed: codes come from HBM)
    j6 = next(j for j, L in enumerate(w.layers) if isinstance(L, synth.FC))
    L6, P6 = w.layers[j6], params[j6]
    x6 = torch.from_numpy(synth.relu_normal((1, L6.Cs), 7)).to(dev)
    D6 = torch.from_numpy(P6["D"]).to(dev)
    c6 = torch.from_numpy(P6["codes"]).to(dev)
    p6 = q.fc_pack_codes(c6, L6.K)
    y6 = torch.empty((1, L6.Ct), device=dev)
    t_byte = event_ms(lambda: q.fc_forward(x6, D6, c6, out=y6), 20)
    t_pack = event_ms(lambda: q.fc_forward(x6, D6, p6, out=y6, Ct=L6.Ct), 20)
    res["model_blob"]["fc6_batch1_us"] = {"byte_codes": round(t_byte * 1e3, 1),
                                          "packed_codes": round(t_pack * 1e3, 1),
                                          "code_bytes": [int(c6.numel()), int(p6.numel())]}

    # ---- quantizer: k-means in every sub-space of every PQ layer, 10 rounds
    rounds = 10
    jobs = []
    for j, L in enumerate(w.layers):
        if isinstance(L, synth.Pool):
            continue
        fan = L.Cs * (L.kh * L.kw if isinstance(L, synth.Conv) else 1)
        shape = (L.Ct, L.Cs, L.kh, L.kw) if isinstance(L, synth.Conv) else (L.Ct, L.Cs)
        Wd = synth.normal(shape, (2.0 / fan) ** 0.5, 150, j)
        M = L.Cs // L.Csp
        if isinstance(L, synth.Conv):
            pts = Wd.reshape(L.Ct, M, L.Csp, L.kh * L.kw).transpose(1, 0, 3, 2).reshape(M, -1, L.Csp)
        else:
            pts = Wd.reshape(L.Ct, M, L.Csp).transpose(1, 0, 2)
        init = np.stack([pts[m][synth.sample_indices(pts.shape[1], L.K, 151, j, m)]
                         for m in range(M)])
        jobs.append((j, L, torch.from_numpy(Wd).to(dev), torch.from_numpy(init).to(dev), Wd, init))

    def quantize_all():
        for j, L, Wt, It, _, _ in jobs:
            if isinstance(L, synth.Conv):
                q.pq_quantize_conv(Wt, L.Csp, L.K, It, rounds)
            else:
                q.pq_quantize_fc(Wt, L.Csp, L.K, It, rounds)

    quantize_all()
    t_q = event_ms(quantize_all, 3, flush_each=False)
    ops = sum((L.Cs // L.Csp) * L.Ct * (L.kh * L.kw if isinstance(L, synth.Conv) else 1) * L.K
              * 3 * L.Csp * (rounds + 1) for _, L, *_ in jobs)
    qres = {"kmeans_alexnet_all_layers_ms": round(t_q, 2), "rounds": rounds,
            "assign_ops": ops, "assign_gops_per_s": round(ops / (t_q / 1e3) / 1e9, 1),
            "note": "assignment: 3 binary32 ops per coordinate per (point, centroid); the time "
                    "includes the sort and the double-precision centroid sums"}
    # error correction on an fc8-shaped layer (4096 -> 1000, C's 4, K 32), 512 vectors
    Ne, Cse, Cte, Cspe, Ke = 512, 4096, 1000, 4, 32
    S = synth.relu_normal((Ne, Cse), 152)
    We = synth.normal((Cte, Cse), (2.0 / Cse) ** 0.5, 153)
    T = (S.astype(np.float64) @ We.astype(np.float64).T).astype(np.float32)
    pe = We.reshape(Cte, Cse // Cspe, Cspe).transpose(1, 0, 2)
    ie = np.stack([pe[m][synth.sample_indices(Cte, Ke, 154, m)] for m in range(Cse // Cspe)])
    D0, c0 = q.pq_quantize_fc(torch.from_numpy(We).to(dev), Cspe, Ke,
                              torch.from_numpy(ie).to(dev), rounds)
    St, Tt = torch.from_numpy(S).to(dev), torch.from_numpy(T).to(dev)
    q.ec_quantize_fc(St, Tt, D0, c0, 1, 2)
    t_ec = event_ms(lambda: q.ec_quantize_fc(St, Tt, D0, c0, 1, 2), 3, flush_each=False)
    qres["ec_fc8_ms"] = round(t_ec, 2)
    qres["ec_setup"] = "N=512 calibration vectors, 1 sweep over 1024 sub-spaces, 2 alternations"
    # error correction of a conv layer (Appendix B), AlexNet conv3 shape with 8
    # calibration images, from the k-means start
    j3, L3, W3t, I3t, W3, I3 = next(t for t in jobs if t[0] == 4)
    Sc = synth.relu_normal((8, L3.Cs, 13, 13), 155)
    Tc = torch.nn.functional.conv2d(torch.from_numpy(Sc).double(), torch.from_numpy(W3).double(),
                                    padding=L3.pad).float()
    Dc0, cc0 = q.pq_quantize_conv(W3t, L3.Csp, L3.K, I3t, rounds)
    Sct, Tct = torch.from_numpy(Sc).to(dev), Tc.to(dev)
    Dc1, cc1 = q.ec_quantize_conv(Sct, Tct, Dc0, cc0, L3.kh, L3.kw, 1, L3.pad, 1, 1)
    t_ecc = event_ms(lambda: q.ec_quantize_conv(Sct, Tct, Dc0, cc0, L3.kh, L3.kw, 1, L3.pad, 1, 1),
                     2, flush_each=False)
    qres["ec_conv3_ms"] = round(t_ecc, 1)

    def rel_err(Dq, cq):
        yq = q.conv_forward(Sct, Dq, cq, L3.kh, L3.kw, 1, L3.pad)
        return float(((yq.double() - Tct.double()) ** 2).sum() / (Tct.double() ** 2).sum())

    qres["ec_conv3_rel_sq_err"] = {"kmeans": round(rel_err(Dc0, cc0), 5),
                                   "error_corrected": round(rel_err(Dc1, cc1), 5)}
    qres["ec_conv3_setup"] = ("8 calibration images 256x13x13 -> 384, C's 4, K 128: one sweep over "
                              "64 sub-spaces, one alternation (128 codeword steps, 9 offset steps)")
    if with_oracle:
        import oracle
        import oracle.ec as oec
        _, L3, W3t, I3t, W3, I3 = next(t for t in jobs if t[0] == 4)   # conv3
        t0 = time.perf_counter()
        oracle.pq_quantize_conv(W3, L3.Csp, L3.K, I3, rounds)
        qres["oracle_kmeans_conv3_s"] = round(time.perf_counter() - t0, 3)
        t3 = event_ms(lambda: q.pq_quantize_conv(W3t, L3.Csp, L3.K, I3t, rounds), 3,
                      flush_each=False)
        qres["kmeans_conv3_ms"] = round(t3, 3)
        t0 = time.perf_counter()
        oec.ec_quantize_fc(S, T, D0.cpu().numpy(), c0.cpu().numpy(), 1, 2)
        qres["oracle_ec_fc8_s"] = round(time.perf_counter() - t0, 3)
    res["quantizer"] = qres

    return res


def build_layers(q, torch, w, params, dev, lut="fp32"):
    """The workload's layers on the device, conv codes packed once (model load)."""
    layers = []
    for L, P in zip(w.layers, params):
        if isinstance(L, synth.Conv):
            codes = q.conv_pack_codes(torch.from_numpy(P["codes"]).to(dev), L.K, L.kh, L.kw)
            layers.append(q.ConvLayer(torch.from_numpy(P["D"]).to(dev), codes,
                                      torch.from_numpy(P["bias"]).to(dev), L.Ct, L.kh, L.kw,
                                      L.stride, L.pad, L.relu, packed=True, lut=lut))
        elif isinstance(L, synth.FC):
            layers.append(q.FCLayer(torch.from_numpy(P["D"]).to(dev),
                                    torch.from_numpy(P["codes"]).to(dev),
                                    torch.from_numpy(P["bias"]).to(dev), L.relu, lut=lut))
        else:
            layers.append(q.PoolLayer(L.k, L.s))
    return layers


def layer_times(q, torch, qlayers, shapes, xin, ws, flush, stream, reps, lut="fp32"):
    """Per-layer ms of a stack launched layer by layer through the C ABI, CUDA
    events between the layers (L2 flushed before each pass; median of reps
    after two untimed passes)."""
    nb = xin.shape[0]
    dev = xin.device
    obufs = [torch.empty((nb, *sout), dtype=torch.float32, device=dev) for (_, sout) in shapes]
    runs = []
    for it in range(reps + 2):
        flush.zero_()
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(len(qlayers) + 1)]
        ev[0].record(stream)
        h = xin
        for j, qL in enumerate(qlayers):
            o = obufs[j]
            if isinstance(qL, q.ConvLayer):
                q.conv_forward(h, qL.D, qL.codes, qL.kh, qL.kw, qL.stride, qL.pad, qL.bias,
                               qL.relu, packed=True, Ct=qL.Ct, out=o, workspace=ws, lut=lut)
            elif isinstance(qL, q.FCLayer):
                q.fc_forward(h.reshape(nb, -1), qL.D, qL.codes, qL.bias, qL.relu,
                             out=o.reshape(nb, -1), workspace=ws, lut=lut)
            else:
                q.maxpool(h, qL.k, qL.s, out=o)
            ev[j + 1].record(stream)
            h = o
        torch.cuda.synchronize(dev)
        if it >= 2:
            runs.append([ev[j].elapsed_time(ev[j + 1]) for j in range(len(qlayers))])
    return [float(np.median([r[j] for r in runs])) for j in range(len(qlayers))]


def measure_configs(q, torch, cm, dev, flush, stream, smem_gbs, hbm_gbs, reps):
    """Every workload at each of its batches (the five configurations of the
    target): the whole stack through qcnn_net_forward (device-resident input,
    L2 flushed before each forward) -- ms, images/s, dense-equivalent GFLOP/s
    and the stack's fraction of the shared-memory roofline -- and per layer
    its ms and the fraction of its stage roofline (stage_rooflines)."""
    cfgs = {}
    for name in sorted(synth.WORKLOADS):
        wk = synth.WORKLOADS[name]
        pk = wk.params()
        lay = build_layers(q, torch, wk, pk, dev)
        in_shape = tuple(wk.in_shape) if len(wk.in_shape) == 3 else (wk.in_shape[0], 1, 1)
        wnet = q.Net(lay, in_shape)
        costs = _layer_costs(wk, cm)
        dense = sum(c.dense_macs for c in costs)
        alg = 4.0 * sum(c.lookups + c.lut_entries for c in costs)
        shapes = wk.shapes()
        per = []
        for B in wk.batches:
            xb = torch.from_numpy(wk.input(B, 3).reshape(B, *in_shape)).to(dev)
            wws = wnet.alloc_workspace(B, dev)
            wout = wnet._out(B, dev)
            for _ in range(3):
                wnet.forward(xb, out=wout, workspace=wws)
            torch.cuda.synchronize(dev)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            ts = []
            for _ in range(reps):
                flush.zero_()
                e0.record(stream)
                wnet.forward(xb, out=wout, workspace=wws)
                e1.record(stream)
                torch.cuda.synchronize(dev)
                ts.append(e0.elapsed_time(e1))
            ms_b = float(np.median(ts))
            xs = xb.reshape(B, *shapes[0][0]) if len(shapes[0][0]) == 3 else xb.reshape(B, -1)
            lws = wnet.alloc_workspace(B, dev)
            stage_ms = layer_times(q, torch, lay, shapes, xs, lws, flush, stream, reps)
            per.append({"batch": B, "ms": round(ms_b, 4), "images_per_s": round(B / (ms_b / 1e3), 1),
                        "dense_equiv_gflops": round(2 * dense * B / (ms_b / 1e3) / 1e9, 1),
                        "frac_smem": round(alg * B / (ms_b / 1e3) / (smem_gbs * 1e9), 4),
                        "stages": stage_rooflines(wk, cm, stage_ms, B, smem_gbs, hbm_gbs)})
        cfgs[name] = per
    # the floor of this timing for a single library call: one launch of the
    # smallest library kernel (a 3x3 max-pool of one 3x3 map), timed the same way
    tiny = torch.zeros((1, 1, 3, 3), dtype=torch.float32, device=dev)
    tout = torch.empty((1, 1, 1, 1), dtype=torch.float32, device=dev)
    for _ in range(3):
        q.maxpool(tiny, 3, 2, out=tout)
    ts = []
    for _ in range(reps):
        flush.zero_()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        q.maxpool(tiny, 3, 2, out=tout)
        e1.record(stream)
        torch.cuda.synchronize(dev)
        ts.append(e0.elapsed_time(e1))
    return {"note": "each workload's whole stack through qcnn_net_forward, device-resident "
                    "input, L2 flushed before every forward; frac_smem = 4 B x (look-ups + "
                    "table entries) per second over the measured shared-memory peak; stages: "
                    "per layer, launched one by one, the fraction of the slower of its "
                    "shared-memory roof and its HBM roof (stage_rooflines); launch_floor_ms: "
                    "one call of the smallest library kernel, timed the same way",
            "launch_floor_ms": round(float(np.median(ts)), 4),
            "workloads": cfgs}


def _layer_costs(w, cm):
    costs = []
    for L, (sin, sout) in zip(w.layers, w.shapes()):
        if isinstance(L, synth.Conv):
            costs.append(cm.conv_cost(L.Cs, L.Ct, sin[1], sin[2], L.kh, L.kw, sout[1], sout[2],
                                      L.Csp, L.K))
        elif isinstance(L, synth.FC):
            costs.append(cm.fc_cost(L.Cs, L.Ct, L.Csp, L.K))
    return costs


def stage_rooflines(w, cm, stage_ms, N, smem_gbs, hbm_gbs):
    """Per-layer fraction of the stage roofline at batch N.  The roof time is
    the slower of two: the algorithmic shared-memory bytes (4 B per look-up and
    per table entry, Table 1 counts) at the shared-memory peak, and the
    algorithmic HBM bytes (input and output activations once, one byte per
    code, the sub-codebooks) at the measured copy bandwidth.  At batch 1 the
    FC layers are HBM-bound (their codes), the conv layers shared-memory
    bound; a max-pool is HBM-bound."""
    out = []
    for j, (L, (sin, sout)) in enumerate(zip(w.layers, w.shapes())):
        t = stage_ms[j] / 1e3
        act = 4.0 * N * (math.prod(sin) + math.prod(sout))
        if isinstance(L, synth.Pool):
            out.append({"layer": j, "kind": "maxpool", "ms": round(stage_ms[j], 4),
                        "bound": "hbm", "frac": round(act / (hbm_gbs * 1e9) / t, 4)})
            continue
        M = L.Cs // L.Csp
        if isinstance(L, synth.Conv):
            c = cm.conv_cost(L.Cs, L.Ct, sin[1], sin[2], L.kh, L.kw, sout[1], sout[2], L.Csp,
                             L.K)
            codes = L.Ct * L.kh * L.kw * M
        else:
            c = cm.fc_cost(L.Cs, L.Ct, L.Csp, L.K)
            codes = L.Ct * M
        t_hbm = (act + codes + 4.0 * M * L.K * L.Csp) / (hbm_gbs * 1e9)
        t_smem = 4.0 * N * (c.lookups + c.lut_entries) / (smem_gbs * 1e9)
        out.append({"layer": j, "kind": L.kind, "ms": round(stage_ms[j], 4),
                    "bound": "hbm" if t_hbm > t_smem else "smem",
                    "frac": round(max(t_hbm, t_smem) / t, 4)})
    return out


def layer_arm(a):
    """One layer of a workload, alone, at --batch: --warmup untimed launches,
    then --steps launches timed with CUDA events (L2 flushed before each).
    For kernel profiles of a single layer (ncu -k / -s / -c)."""
    import torch

    import paper_1512_06473_gb300 as q
    name, idx = a.layer.split(":")
    idx = int(idx)
    dev = torch.device("cuda", 0)
    w = synth.WORKLOADS[name]
    params = w.params()
    lay = build_layers(q, torch, w, params, dev)
    qL, (sin, sout) = lay[idx], w.shapes()[idx]
    N = a.batch
    x = torch.from_numpy(synth.relu_normal((N, *sin), 0, idx)).to(dev)
    y = torch.empty((N, *sout), dtype=torch.float32, device=dev)
    ws = torch.empty(1 << 30, dtype=torch.uint8, device=dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)

    def run():
        if isinstance(qL, q.ConvLayer):
            q.conv_forward(x, qL.D, qL.codes, qL.kh, qL.kw, qL.stride, qL.pad, qL.bias, qL.relu,
                           packed=True, Ct=qL.Ct, out=y, workspace=ws)
        elif isinstance(qL, q.FCLayer):
            q.fc_forward(x.reshape(N, -1), qL.D, qL.codes, qL.bias, qL.relu,
                         out=y.reshape(N, -1), workspace=ws)
        else:
            q.maxpool(x, qL.k, qL.s, out=y)

    for _ in range(a.warmup):
        run()
    ts = []
    for _ in range(a.steps):
        flush.zero_()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        run()
        e1.record()
        torch.cuda.synchronize(dev)
        ts.append(e0.elapsed_time(e1))
    plan = None
    if isinstance(qL, q.ConvLayer):
        plan = q.conv_plan(N, sin[0], sin[1], sin[2], qL.Ct, qL.kh, qL.kw, qL.stride, qL.pad,
                           w.layers[idx].Csp, w.layers[idx].K)
    elif isinstance(qL, q.FCLayer):
        L = w.layers[idx]
        plan = q.fc_plan(N, L.Cs, L.Ct, L.Csp, L.K)
    print(json.dumps({"layer": a.layer, "batch": N, "ms_median": float(np.median(ts)),
                      "steps": a.steps, "plan": plan}), flush=True)
    return 0


def main():
    a = parse()
    if a.impl == "reference":
        return reference_arm(a)
    if a.layer:
        return layer_arm(a)

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))

    # The CPU-baseline pool is spawned before the first GPU call.
    pool = None
    cores = min(os.cpu_count() or 1, 16)
    if rank == 0 and world == 1 and not a.no_cpu_baseline:
        pool = oracle_pool(cores, a.batch)

    import torch
    import torch.distributed as dist

    import paper_1512_06473_gb300 as q
    from paper_1512_06473_gb300 import costmodel as cm

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)

    w = synth.WORKLOADS[WORKLOAD]
    N = a.batch
    params = w.params()
    x_host = torch.from_numpy(w.input(N, rank)).pin_memory()
    x = x_host.to(dev)

    # model load: codes re-laid out once, outside the timed region
    shapes = w.shapes()

    def make_layers(lut):
        layers = []
        for L, P in zip(w.layers, params):
            if isinstance(L, synth.Conv):
                codes = q.conv_pack_codes(torch.from_numpy(P["codes"]).to(dev), L.K, L.kh, L.kw)
                layers.append(q.ConvLayer(torch.from_numpy(P["D"]).to(dev), codes,
                                          torch.from_numpy(P["bias"]).to(dev), L.Ct, L.kh, L.kw,
                                          L.stride, L.pad, L.relu, packed=True, lut=lut))
            elif isinstance(L, synth.FC):
                layers.append(q.FCLayer(torch.from_numpy(P["D"]).to(dev),
                                        torch.from_numpy(P["codes"]).to(dev),
                                        torch.from_numpy(P["bias"]).to(dev), L.relu, lut=lut))
            else:
                layers.append(q.PoolLayer(L.k, L.s))
        return layers

    layers = make_layers("fp32")
    net = q.Net(layers, tuple(w.in_shape))
    ws = net.alloc_workspace(N, dev)
    out = net._out(N, dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)  # > 129 MB L2
    stream = torch.cuda.current_stream(dev)

    def step():
        net.forward(x, out=out, workspace=ws)

    for _ in range(max(a.warmup, 3)):
        step()
    torch.cuda.synchronize(dev)

    clocks = ClockSampler(local)
    clocks.start()
    l0 = q.launch_count()
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(a.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(a.steps)]
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    t0 = clocks.mark()
    for i in range(a.steps):
        flush.zero_()
        starts[i].record(stream)
        step()
        ends[i].record(stream)
    torch.cuda.synchronize(dev)
    t1 = clocks.mark()
    if world > 1:
        dist.barrier()
    launches = q.launch_count() - l0
    clk = clocks.stop(t0, t1)
    ms = sum(s.elapsed_time(e) for s, e in zip(starts, ends))
    if world > 1:
        ms = max_over_ranks(ms, dev)
    ms_per_step = ms / a.steps
    value = job_throughput(N, world, a.steps, ms / 1e3)

    # ---- per-stage timing: the same layers launched one by one, events between
    bufs = [torch.empty((N, *sout), dtype=torch.float32, device=dev) for (sin, sout) in shapes]
    lws = torch.empty(ws.numel(), dtype=torch.uint8, device=dev)

    def stage_times(qlayers, lut, xin=None, obufs=None):
        xin = x if xin is None else xin
        obufs = bufs if obufs is None else obufs
        nb = xin.shape[0]
        stage_ms = [0.0] * len(qlayers)
        for it in range(a.steps + 2):
            flush.zero_()
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(len(qlayers) + 1)]
            ev[0].record(stream)
            h = xin
            for j, qL in enumerate(qlayers):
                o = obufs[j]
                if isinstance(qL, q.ConvLayer):
                    q.conv_forward(h, qL.D, qL.codes, qL.kh, qL.kw, qL.stride, qL.pad, qL.bias,
                                   qL.relu, packed=True, Ct=qL.Ct, out=o, workspace=lws, lut=lut)
                elif isinstance(qL, q.FCLayer):
                    q.fc_forward(h.reshape(nb, -1), qL.D, qL.codes, qL.bias, qL.relu,
                                 out=o.reshape(nb, -1), workspace=lws, lut=lut)
                else:
                    q.maxpool(h, qL.k, qL.s, out=o)
                ev[j + 1].record(stream)
                h = o
            torch.cuda.synchronize(dev)
            if it >= 2:
                for j in range(len(qlayers)):
                    stage_ms[j] += ev[j].elapsed_time(ev[j + 1])
        return [t / a.steps for t in stage_ms]

    peaks = load_peaks()
    sm_max = float(peaks.get("sm_max_mhz") or 2070.0)
    nsm = torch.cuda.get_device_properties(dev).multi_processor_count
    # shared-memory peak: 128 B per wavefront x the wavefronts per SM per cycle
    # a conflict-free 16-byte-per-lane load stream sustains on this GPU,
    # measured now (qcnn_smem_load_rate) x SMs x the maximum SM clock
    smem_wpc = {"lds128": round(q.smem_load_rate(16), 4), "lds32": round(q.smem_load_rate(4), 4)}
    smem_peak_gbs = nsm * 128 * smem_wpc["lds128"] * sm_max * 1e6 / 1e9

    def stage_report(stage_ms, entry_bytes):
        """Per-layer ms and shared-memory roofline fraction; algorithmic bytes =
        entry_bytes x (look-ups + table entries) (Table 1 counts)."""
        stages, dense = [], 0.0
        for j, (L, (sin, sout)) in enumerate(zip(w.layers, shapes)):
            if isinstance(L, synth.Conv):
                c = cm.conv_cost(L.Cs, L.Ct, sin[1], sin[2], L.kh, L.kw, sout[1], sout[2], L.Csp,
                                 L.K)
            elif isinstance(L, synth.FC):
                c = cm.fc_cost(L.Cs, L.Ct, L.Csp, L.K)
            else:
                stages.append({"layer": j, "kind": "maxpool", "ms": round(stage_ms[j], 4)})
                continue
            dense += c.dense_macs
            alg_bytes = entry_bytes * (c.lookups + c.lut_entries) * N
            ach = alg_bytes / (stage_ms[j] / 1e3) / 1e9
            stages.append({"layer": j, "kind": L.kind, "ms": round(stage_ms[j], 4),
                           "lookups": c.lookups * N, "lut_entries": c.lut_entries * N,
                           "smem_alg_GBs": round(ach, 1),
                           "frac_smem": round(ach / smem_peak_gbs, 4)})
        return stages, dense

    stages, dense_macs = stage_report(stage_times(layers, "fp32"), 4.0)
    dom = max((s for s in stages if s["kind"] != "maxpool"), key=lambda s: s["ms"])
    dom_alg = 4.0 * (dom["lookups"] + dom["lut_entries"])
    roofline = {
        "bound": "smem", "kernel": f"layer {dom['layer']} ({dom['kind']})",
        "achieved": round(dom_alg / (dom["ms"] / 1e3) / 1e9, 1),
        "peak": round(smem_peak_gbs, 1), "unit": "GB/s",
        "frac": round(dom_alg / (dom["ms"] / 1e3) / 1e9 / smem_peak_gbs, 4),
        "traffic": recorded_traffic(WORKLOAD, N, dom["layer"]),
        "traffic_note": "DRAM read+write bytes per launch (ncu, profiles/dram_traffic.txt); "
                        "the kernel's algorithmic traffic is shared-memory, not DRAM",
        "peak_basis": (f"{nsm} SMs x 128 B x {smem_wpc['lds128']} wavefronts/clk "
                       f"(measured now: conflict-free 16-byte shared loads, qcnn_smem_load_rate; "
                       f"4-byte loads: {smem_wpc['lds32']}) x {sm_max:.0f} MHz max SM clock"),
        "alg_bytes_per_launch": dom_alg,
    }

    # ---- end to end through qcnn_net_forward_host (pinned host buffers)
    ws_h = net.alloc_workspace(N, dev, host_io=True)
    y_host = torch.empty(tuple(out.shape), dtype=torch.float32).pin_memory()
    for _ in range(2):
        net.forward_host(x_host, y_host, ws_h)
    e2e_t = 0.0
    for _ in range(a.steps):
        flush.zero_()
        torch.cuda.synchronize(dev)
        t = time.perf_counter()
        net.forward_host(x_host, y_host, ws_h)
        e2e_t += time.perf_counter() - t
    if world > 1:
        e2e_t = max_over_ranks(e2e_t, dev)
    e2e = {"value": job_throughput(N, world, a.steps, e2e_t), "unit": "images/s",
           "h2d_bytes_per_step": x_host.numel() * 4, "d2h_bytes_per_step": y_host.numel() * 4}

    # ---- batch 1 latency: plain launches, and one CUDA graph of the whole stack
    x1 = x[:1].contiguous()

    def batch1(bnet):
        ws1 = bnet.alloc_workspace(1, dev)
        o1 = bnet._out(1, dev)
        for _ in range(5):
            bnet.forward(x1, out=o1, workspace=ws1)
        torch.cuda.synchronize(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

        def median_ms(fn):
            lat = []
            for _ in range(20):
                flush.zero_()
                e0.record(stream)
                fn()
                e1.record(stream)
                torch.cuda.synchronize(dev)
                lat.append(e0.elapsed_time(e1))
            return float(np.median(lat))

        res = {"latency_ms": round(median_ms(lambda: bnet.forward(x1, out=o1, workspace=ws1)), 4)}
        res["images_per_s"] = round(1e3 / res["latency_ms"], 1)
        try:
            g = torch.cuda.CUDAGraph()
            side = torch.cuda.Stream(dev)
            side.wait_stream(stream)
            with torch.cuda.stream(side):
                with torch.cuda.graph(g, stream=side):
                    bnet.forward(x1, out=o1, workspace=ws1)
            stream.wait_stream(side)
            g.replay()
            torch.cuda.synchronize(dev)
            res["graph_latency_ms"] = round(median_ms(g.replay), 4)
        except Exception as e:  # capture refused: report it, keep the plain number
            res["graph_error"] = f"{type(e).__name__}: {e}"[:200]
        return res

    b1 = batch1(net)
    bufs1 = [torch.empty((1, *sout), dtype=torch.float32, device=dev) for (sin, sout) in shapes]
    b1["stage_ms"] = [round(t, 4) for t in stage_times(layers, "fp32", x1, bufs1)]
    hbm_gbs = float(peaks.get("hbm_gbs") or 6800.0)
    b1["stages"] = stage_rooflines(w, cm, b1["stage_ms"], 1, smem_peak_gbs, hbm_gbs)
    b1["roofline_note"] = (f"per stage: the slower of shared-memory bytes at {smem_peak_gbs:.0f} "
                           f"GB/s and HBM bytes at {hbm_gbs:.0f} GB/s (measured copy)")

    # ---- every workload of the target at its batches, per layer (GPU)
    configs = measure_configs(q, torch, cm, dev, flush, stream, smem_peak_gbs, hbm_gbs,
                              max(5, a.steps // 3))

    extras = {}
    if not a.no_extras:
        extras = extra_measurements(a, q, torch, w, params, x, out, flush, stream, dev, N,
                                    batch1, cm, rank == 0 and world == 1)

    cpu = None
    if pool is not None:
        sample = a.cpu_sample or cores
        dt = time_oracle(pool, cores, sample, N)
        cfg_oracle = oracle_configs(pool, cores)
        pool.close()
        cpu = {"value": sample / dt, "unit": "images/s", "cores": cores, "kind": "oracle",
               "sample": f"{sample} images of the batch-{N} workload, one per spawned process, "
                         f"float64 C oracle, host {_cpu_info()}, {dt:.1f} s wall",
               "configs": cfg_oracle,
               "configs_note": "every workload: its smallest batch on one core alone "
                               "(single_thread), and for workloads with a large batch, "
                               "images on all cores (all_cores); same float64 C oracle"}

    if world > 1:
        dist.destroy_process_group()
    if rank != 0:
        return 0
    line = {
        "metric": METRIC, "value": round(value, 1), "unit": "images/s", "n_gpus": world,
        "steps": a.steps, "warmup": max(a.warmup, 3), "ms_per_step": round(ms_per_step, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic (seeded images, random-init codebooks/codes/biases)",
        "config": {"workload": WORKLOAD, "global_batch": N * world, "per_gpu_batch": N,
                   "image": "3x227x227", "parallelism": f"replicas x{world}",
                   "l2": "flushed (256 MB write) before every timed step",
                   "codes": "packed once at model load (outside the timed region)"},
        "dense_equiv_gflops": round(2 * dense_macs * value / 1e9, 1),
        "batch1": b1,
        "roofline": roofline, "stages": stages, "configs": configs, **extras,
        "cpu_baseline": cpu, "e2e": {k: (round(v, 1) if isinstance(v, float) else v)
                                     for k, v in e2e.items()},
        "gpu_launches": int(launches), "clocks": clk,
    }
    print(json.dumps(line), flush=True)
    return 0


if __name__ == "__main__":
    sys.exit(main())
