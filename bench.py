"""Benchmark of batched TFHE programmable bootstrapping on GB300.

One step = one rosetta_pbs_batch call over the whole batch (modulus switch,
blind rotation, sample extraction, key switch) with keys and inputs resident
in HBM.  Default workload: the standard parameter set (n=742, k=1, N=2048,
PBS base 2^23 x 1, KS base 2^3 x 5) on a batch of 4096 ciphertexts with a
4-bit GELU LUT.

Prints one JSON line (rank 0).  `--impl reference` times the CPU oracle on
the host cores instead (the reference arm: a deliberately plain program).

`--path lookup` measures the encrypted segmented lookup instead (the
lookup protocol's Steps 2 and 3 composed from plaintext products, blind
rotations of GLWE test polynomials, a key switch and RLWE traces) on the
same ring, four segments, one line of its own; `--path multi_lut` the PBS
with a LUT per ciphertext (four LUTs in one launch); `--path peaks` the
integer issue rates of the GPU (operations per clock per SM for IADD3, LOP3,
IMAD, IMAD.HI, IMAD.WIDE, an IMAD+IADD3 mix, the NTT butterfly, and the
butterfly that primes near 2^31 would need).
"""

from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import workload as W  # noqa: E402

METRIC = "PBS/sec (blind rotate + key switch) on 1 GB300; fraction of roofline"
UNIT = "PBS/s"


def describe(p, batch):
    return (f"{p.name}: n={p.n} k={p.k} N={p.N} PBS base 2^{p.pbs_base_log} x {p.pbs_level}, "
            f"KS base 2^{p.ks_base_log} x {p.ks_level}, {p.msg_bits}-bit LUT {p.lut[0]}, batch {batch}")


# ---------------------------------------------------------------------------- op counts

def min_primes(p) -> int:
    """Smallest number of 31-bit primes whose product exceeds twice the
    largest integer value of an external-product coefficient."""
    bits = 63 + (p.pbs_base_log - 1) + math.log2((p.k + 1) * p.pbs_level * p.N) + 1
    return math.ceil(bits / 31)


def int_ops_per_pbs(p):
    """Algorithmic 32-bit integer operations of one PBS: (blind rotation,
    key switch).  Counting convention: NTT butterflies 8 ops, pointwise
    multiply-accumulate 6, CRT 10 per prime, decomposition 6 per level,
    rotation/accumulate 4, per coefficient; key switch 3 per digit x word."""
    P = min_primes(p)
    k1, l, N = p.k + 1, p.pbs_level, p.N
    per_cmux = ((k1 * l + k1) * P * (N // 2) * int(math.log2(N)) * 8 + k1 * l * k1 * P * N * 6
                + k1 * N * 10 * P + k1 * N * l * 6 + k1 * N * 4)
    ks = p.kN * p.ks_level * (p.n + 1) * 3 + p.kN * p.ks_level * 6
    return per_cmux * p.n, ks


def _ntt_ops(N: int) -> int:
    return (N // 2) * int(math.log2(N)) * 8


def _primes_for(bits: float) -> int:
    return math.ceil(bits / 31)


def int_ops_key_switch_step(N: int, base_log: int, rows: int, outs: int = 2) -> int:
    """One GLWE key switch (trace step) or plaintext product: `rows` digit
    polynomials times `outs` key components, same convention as above."""
    P = _primes_for(63 + (base_log - 1) + math.log2(rows * N) + 1)
    return ((rows + outs) * P * _ntt_ops(N) + rows * outs * P * N * 6 + outs * N * 10 * P
            + N * rows * 6 + outs * N * 4)


def int_ops_per_lookup(p, n_seg: int, t_base_log: int, t_level: int) -> dict:
    """Per encrypted lookup: n_seg + 2 blind rotations, one key switch,
    n_seg + 1 traces (log2 N key-switch steps each), n_seg + 2 plaintext
    products (exact 16 x 4 gadget on both components: 8 rows; per output
    only 4 are nonzero, which bounds the primes)."""
    br, ks = int_ops_per_pbs(p)
    logN = int(math.log2(p.N))
    tr = logN * int_ops_key_switch_step(p.N, t_base_log, t_level)
    P = _primes_for(63 + 15 + math.log2(4 * p.N) + 1)
    pm = (8 + 2) * P * _ntt_ops(p.N) + 8 * 2 * P * p.N * 6 + 2 * p.N * 10 * P + 2 * p.N * 4 * 6 + 2 * p.N * 4
    return {"blind_rotation": (n_seg + 2) * br, "key_switch": ks, "trace": (n_seg + 1) * tr,
            "plaintext_mul": (n_seg + 2) * pm, "monomial": n_seg * 2 * p.N * 2}


def ks_tensor_limbs(p, batch) -> int:
    """Limbs per key word of the tensor-core key switch the library takes for
    this batch (8 or 16), or 0 when it takes the CUDA-core kernel: batches of
    256 and more, digits that bf16 holds, fp32 sums below 2^24."""
    K = p.kN * p.ks_level
    if batch < 256 or p.ks_base_log > 8 or K % 64:
        return 0
    for limbs in (8, 16):
        if 2 ** (p.ks_base_log - 1) * (2 ** (64 // limbs) - 1) * K < 2 ** 24:
            return limbs
    return 0


def ks_tensor_flops(p, batch, limbs) -> float:
    """Dense bf16 flops of the tensor-core key switch as launched: 128-row by
    256-column output tiles over K = kN l."""
    K = p.kN * p.ks_level
    rows = -(-batch // 128) * 128
    cols = -(-(p.n + 1) * limbs // 256) * 256
    return 2.0 * rows * K * cols


TRAFFIC_SUMMARY = os.path.join(ROOT, "profiles", "blind_rotate_standard_b4096_dram.txt")


def measured_traffic(p, batch):
    """DRAM bytes (read + write) of one blind-rotation launch from the
    committed ncu summary, or None when the summary is for another workload
    or the kernel sources changed since it was captured."""
    import hashlib
    try:
        kv = dict(line.strip().split("=", 1) for line in open(TRAFFIC_SUMMARY)
                  if "=" in line and not line.startswith("#"))
    except OSError:
        return None
    if kv.get("config") != p.name or int(kv.get("batch", -1)) != batch:
        return None
    h = hashlib.sha256()
    for f in kv["sources"].split(","):
        h.update(open(os.path.join(ROOT, "paper_2609_16915_gb300", "csrc", f), "rb").read())
    if h.hexdigest() != kv.get("sources_sha256"):
        return None
    return int(kv["dram_bytes_read"]) + int(kv["dram_bytes_write"])


def peaks():
    try:
        return json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except OSError:
        return {}


# ---------------------------------------------------------------------------- integer issue rates

INT_OPS = {0: "IADD3", 1: "LOP3", 2: "IMAD", 3: "IMAD.HI", 4: "IMAD.WIDE", 5: "IMAD+IADD3", 6: "butterfly",
           7: "butterfly_p31"}


def measure_int_rates(torch, dev, iters: int = 16384) -> dict:
    """32-bit integer operations retired per clock per SM for each class
    (libintpeaks.so: eight independent inline-PTX chains per thread, 4 CTAs
    of 512 threads per SM).  The rate uses the SM clock the kernels
    themselves saw (clock64 over %globaltimer), so it does not depend on the
    clock the run happened to get; `mhz` reports that clock."""
    import ctypes
    from paper_2609_16915_gb300 import build as B
    L = ctypes.CDLL(B.build_peaks())
    L.intpeak_launch.argtypes = [ctypes.c_int, ctypes.c_uint32, ctypes.c_uint32, ctypes.c_uint32, ctypes.c_void_p,
                                 ctypes.c_void_p, ctypes.c_void_p]
    L.intpeak_ops_per_iter.restype = ctypes.c_uint32
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    ctas, threads = 4 * sms, 512
    sink = torch.zeros(1, dtype=torch.int32, device=dev)
    stamps = torch.zeros(2 * ctas, dtype=torch.int64, device=dev)
    stream = torch.cuda.current_stream(dev)
    out = {}
    for op, name in INT_OPS.items():
        # one untimed launch, then the timed one
        st = L.intpeak_launch(op, ctas, threads, iters, sink.data_ptr(), stamps.data_ptr(), stream.cuda_stream)
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        st = st or L.intpeak_launch(op, ctas, threads, iters, sink.data_ptr(), stamps.data_ptr(), stream.cuda_stream)
        b.record(stream)
        torch.cuda.synchronize(dev)
        if st != 0:
            raise RuntimeError(f"intpeak_launch({name}) failed: cudaError {st}")
        ms = a.elapsed_time(b)
        st = stamps.cpu().numpy().reshape(ctas, 2).astype(np.float64)
        mhz = float(np.median(st[:, 0] / st[:, 1]) * 1e3)
        ops = float(L.intpeak_ops_per_iter(op)) * iters * threads * ctas
        out[name] = {"per_clk_per_sm": ops / (ms * 1e-3 * sms * mhz * 1e6), "mhz": mhz, "ms": ms}
    out["sms"] = sms
    return out


# ---------------------------------------------------------------------------- clocks

class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *a):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 8:
                continue
            try:
                sm.append(float(f[0]))
                mx = float(f[1])
            except ValueError:
                continue
            for name, v in zip(names, f[4:8]):
                if v.lower() == "active":
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------------------- oracle (CPU) timing

def oracle_pbs_rate(p, count, threads=None, seed=0):
    """PBS/s of the CPU oracle on `count` ciphertexts with uniform-word keys."""
    import oracle as O
    bsk, ksk = W.uniform_keys(p)
    lwe = W.uniform_ciphertexts(p, count, sub=1000 + seed)
    lut = W.lut_torus(p)
    t = threads or O.default_threads()
    t0 = time.perf_counter()
    O.pbs_batch(p, bsk, ksk, lwe, lut, threads=t)
    dt = time.perf_counter() - t0
    return count / dt, dt, t


def run_reference(args, p, batch):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    import oracle as O
    O.build()
    cores = O.default_threads()
    sample = max(1, min(batch, cores))
    for _ in range(args.warmup):
        oracle_pbs_rate(p, 1, threads=1)
    rates, times = [], []
    for s in range(args.steps):
        r, dt, t = oracle_pbs_rate(p, sample, threads=cores, seed=s)
        rates.append(r)
        times.append(dt)
    value = sample * len(times) / sum(times)
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * sum(times) / len(times),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u64", "data": "synthetic",
        "config": {"workload": describe(p, batch), "batch": batch, "keys": "uniform words"},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": f"{sample} ciphertexts of the workload per step (schoolbook CPU oracle)"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------------------- lookup path

LOOKUP_METRIC = "encrypted segmented lookups/sec (lookup protocol Steps 2-3, 4 segments) on 1 GB300"
LOOKUP_SEGMENTS, LOOKUP_TRACE = 4, (16, 4)


def run_lookup(args, p, batch, torch, dev, R, clock_sampler):
    """Throughput of rosetta_segmented_lookup_batch on `batch` ciphertexts,
    plus each component entry point timed alone on the same batch."""
    n_seg = LOOKUP_SEGMENTS
    tb, tl = LOOKUP_TRACE
    g = np.random.default_rng(p.seed)

    def d(a):
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int64)).to(dev)

    bsk, ksk = W.uniform_keys(p)
    ctx = R.Context(p, device=dev.index or 0)
    ctx.upload_bsk(d(bsk))
    ctx.upload_ksk(d(ksk))
    del bsk, ksk
    steps = int(math.log2(p.N))
    ctx.upload_trace_keys(d(W.uniform_u64((steps, tl, 2, p.N), W.rng(p.seed, "sample", 300))), tb, tl)
    tables = (g.integers(-2**40, 2**40, size=p.N, dtype=np.int64), W.uniform_u64((p.N,), W.rng(p.seed, "sample", 301)),
              g.integers(-2**40, 2**40, size=(n_seg, p.N), dtype=np.int64),
              W.uniform_u64((n_seg, p.N), W.rng(p.seed, "sample", 302)))
    ctx.upload_lookup_table(*tables)
    glwe = d(W.uniform_u64((batch, 2, p.N), W.rng(p.seed, "sample", 303)))
    lwe = d(W.uniform_ciphertexts(p, batch, sub=7))
    out = torch.empty((batch, 2, p.N), dtype=torch.int64, device=dev)
    tmp = torch.empty((batch, 2, p.N), dtype=torch.int64, device=dev)
    stream = torch.cuda.current_stream(dev)
    flush = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.int32, device=dev)
    for _ in range(max(3, args.warmup)):
        ctx.segmented_lookup_batch(glwe, lwe, out, stream)
    ctx.sync_status(stream)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    torch.cuda.synchronize(dev)
    with clock_sampler(dev.index or 0) as clk:
        for s in range(args.steps):
            flush.zero_()
            ev[s][0].record(stream)
            ctx.segmented_lookup_batch(glwe, lwe, out, stream)
            ev[s][1].record(stream)
        torch.cuda.synchronize(dev)
    ctx.sync_status(stream)
    total_ms = sum(a.elapsed_time(b) for a, b in ev)
    value = batch * args.steps / (total_ms / 1e3)

    def timed(fn, reps=3):
        e = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(reps)]
        for i in range(reps):
            flush.zero_()
            e[i][0].record(stream)
            fn()
            e[i][1].record(stream)
        ctx.sync_status(stream)
        return statistics.mean(a.elapsed_time(b) for a, b in e)

    br_ms = timed(lambda: ctx.blind_rotate_glwe_batch(lwe, glwe, tmp, stream))
    tr_ms = timed(lambda: ctx.trace_batch(glwe, tmp, stream))
    ops = int_ops_per_lookup(p, n_seg, tb, tl)
    br_ops = int_ops_per_pbs(p)[0]
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    sm_max = peaks().get("sm_max_mhz", 2070.0)
    alu_peak = sms * 128 * sm_max * 1e6 / 1e12
    achieved = br_ops * batch / (br_ms / 1e3) / 1e12
    path_achieved = sum(ops.values()) * batch * args.steps / (total_ms / 1e3) / 1e12
    line = {
        "metric": LOOKUP_METRIC, "value": value, "unit": "lookups/s", "n_gpus": 1, "steps": args.steps,
        "warmup": max(3, args.warmup), "ms_per_step": total_ms / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "u64", "data": "synthetic",
        "config": {"workload": f"segmented lookup, {n_seg} segments, ring of {describe(p, batch)}, "
                               f"trace gadget 2^{tb} x {tl}", "batch": batch,
                   "l2": "flushed between steps (256 MB write)", "keys": "uniform words, resident"},
        "roofline": {"bound": "alu", "kernel": "blind_rotate_kernel (GLWE test polynomials)", "achieved": achieved,
                     "peak": alu_peak, "unit": "Tops/s (int32)", "frac": achieved / alu_peak, "traffic": None,
                     "kernel_ms": br_ms, "trace_ms": tr_ms,
                     "path_ops_per_lookup": ops, "path_achieved": path_achieved,
                     "path_frac": path_achieved / alu_peak},
        "gpu_launches": (4 * n_seg + 6) * args.steps,
        "clocks": clk.summary(),
    }
    return line


# ---------------------------------------------------------------------------- many-LUT path

MULTI_METRIC = "PBS/sec with a LUT per ciphertext (4 LUTs in one launch) on 1 GB300"


def run_multi_lut(args, p, batch, torch, dev, R, clock_sampler):
    """Throughput of rosetta_pbs_batch_multi_lut: four LUTs (the workload's
    and three shifted copies) assigned round-robin to the ciphertexts."""
    def d(a):
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int64)).to(dev)

    bsk, ksk = W.uniform_keys(p)
    ctx = R.Context(p, device=dev.index or 0, max_batch=batch)
    ctx.upload_bsk(d(bsk))
    ctx.upload_ksk(d(ksk))
    del bsk, ksk
    codes = W.lut_codes(p)
    luts = d(np.stack([W.lut_torus(p, np.roll(codes, r)) for r in range(4)]))
    idx = torch.from_numpy((np.arange(batch) % 4).astype(np.int32)).to(dev)
    lwe = d(W.uniform_ciphertexts(p, batch, sub=9))
    out = torch.empty((batch, p.n + 1), dtype=torch.int64, device=dev)
    stream = torch.cuda.current_stream(dev)
    flush = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.int32, device=dev)
    for _ in range(max(3, args.warmup)):
        ctx.pbs_batch_multi_lut(lwe, luts, idx, out, stream)
    ctx.sync_status(stream)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    torch.cuda.synchronize(dev)
    with clock_sampler(dev.index or 0) as clk:
        for s_ in range(args.steps):
            flush.zero_()
            ev[s_][0].record(stream)
            ctx.pbs_batch_multi_lut(lwe, luts, idx, out, stream)
            ev[s_][1].record(stream)
        torch.cuda.synchronize(dev)
    ctx.sync_status(stream)
    total_ms = sum(a.elapsed_time(b) for a, b in ev)
    value = batch * args.steps / (total_ms / 1e3)
    br_ops, ks_ops = int_ops_per_pbs(p)
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    alu_peak = sms * 128 * peaks().get("sm_max_mhz", 2070.0) * 1e6 / 1e12
    achieved = br_ops * batch * args.steps / (total_ms / 1e3) / 1e12
    line = {
        "metric": MULTI_METRIC, "value": value, "unit": "PBS/s", "n_gpus": 1, "steps": args.steps,
        "warmup": max(3, args.warmup), "ms_per_step": total_ms / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "u64", "data": "synthetic",
        "config": {"workload": describe(p, batch) + ", 4 LUTs round-robin", "batch": batch,
                   "l2": "flushed between steps (256 MB write)", "keys": "uniform words, resident"},
        "roofline": {"bound": "alu", "kernel": "blind_rotate_kernel + key switch (whole step)", "achieved": achieved,
                     "peak": alu_peak, "unit": "Tops/s (int32)", "frac": achieved / alu_peak, "traffic": None},
        "gpu_launches": (3 if ks_tensor_limbs(p, batch) else 2) * args.steps,
        "clocks": clk.summary(),
    }
    return line


# ---------------------------------------------------------------------------- other workloads, same run

class _Steps:
    """argparse-like holder for the short runs of the other workloads."""

    def __init__(self, steps, warmup):
        self.steps, self.warmup = steps, warmup


class _NoClock:
    def __init__(self, *_):
        pass

    def __enter__(self):
        return self

    def __exit__(self, *_):
        pass

    def summary(self):
        return None


def butterfly_rate(rates, primes):
    """Measured butterflies per clock per SM of the butterfly the blind
    rotation runs: the lazy one of the 28-bit primes (five instructions) or
    the one of the 31-bit primes (nine)."""
    return rates["butterfly_p31"]["per_clk_per_sm"] / 9.0 if primes == 3 else rates["butterfly"]["per_clk_per_sm"] / 5.0


def kernel_name(primes):
    return "blind_rotate3_kernel (3 primes)" if primes == 3 else "blind_rotate_kernel (4 primes)"


def measure_other_config(name, torch, dev, R, steps, warmup, sms, sm_max, rates):
    """PBS/s of another parameter set at its full batch (uniform-word keys and
    ciphertexts resident, L2 flushed between steps), the blind rotation timed
    alone, and its fractions of the two peaks."""
    p = W.CONFIGS[name]
    batch = p.batch

    def d(a):
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int64)).to(dev)

    bsk, ksk = W.uniform_keys(p)
    ctx = R.Context(p, device=dev.index or 0, max_batch=batch)
    ctx.upload_bsk(d(bsk))
    ctx.upload_ksk(d(ksk))
    del bsk, ksk
    lwe = d(W.uniform_ciphertexts(p, batch, sub=1))
    lut = d(W.lut_torus(p))
    out = torch.empty((batch, p.n + 1), dtype=torch.int64, device=dev)
    big = torch.empty((batch, p.kN + 1), dtype=torch.int64, device=dev)
    stream = torch.cuda.current_stream(dev)
    flush = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.int32, device=dev)
    for _ in range(warmup):
        ctx.pbs_batch(lwe, lut, out, stream)
    ctx.sync_status(stream)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    for a, b in ev:
        flush.zero_()
        a.record(stream)
        ctx.pbs_batch(lwe, lut, out, stream)
        b.record(stream)
    flush.zero_()
    a1, b1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a1.record(stream)
    ctx.blind_rotate_extract_batch(lwe, lut, big, stream)
    b1.record(stream)
    ctx.sync_status(stream)
    ms = sum(a.elapsed_time(b) for a, b in ev) / steps
    br_ms = a1.elapsed_time(b1)
    br_ops, _ = int_ops_per_pbs(p)
    achieved = br_ops * batch / (br_ms / 1e3) / 1e12
    primes = ctx.ntt_primes()
    bfly_per_clk = butterfly_rate(rates, primes)
    ctx.close()
    del lwe, out, big, flush
    torch.cuda.empty_cache()
    return {"workload": describe(p, batch), "value": batch / (ms / 1e3), "unit": UNIT, "ms_per_step": ms,
            "steps": steps, "warmup": warmup, "kernel": kernel_name(primes), "blind_rotation_ms": br_ms,
            "achieved_tops": achieved, "frac": achieved / (sms * 128 * sm_max * 1e6 / 1e12),
            "frac_of_butterfly_rate_peak": achieved / (bfly_per_clk * 8 * sms * sm_max * 1e6 / 1e12),
            "butterflies_per_clk_per_sm": round(bfly_per_clk, 2)}


# ---------------------------------------------------------------------------- GPU arm

def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", default="standard", choices=sorted(W.CONFIGS))
    ap.add_argument("--batch", type=int, default=0, help="override the workload's batch")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-other", action="store_true",
                    help="skip the short runs of the other parameter sets and paths that follow the headline")
    ap.add_argument("--cpu-sample", type=int, default=0, help="oracle sample size (default: three per host core)")
    ap.add_argument("--path", default="pbs", choices=["pbs", "lookup", "multi_lut", "peaks"])
    args = ap.parse_args()
    p = W.CONFIGS[args.config]
    batch = args.batch or p.batch
    if args.impl == "reference":
        return run_reference(args, p, batch)
    if args.path in ("lookup", "multi_lut", "peaks"):
        import torch
        import paper_2609_16915_gb300 as R
        R.load()
        dev = torch.device("cuda", 0)
        torch.cuda.set_device(dev)
        if args.path == "peaks":
            with ClockSampler(0) as clk:
                rates = measure_int_rates(torch, dev)
            print(json.dumps({"metric": "32-bit integer operations per clock per SM", "rates": rates,
                              "clocks": clk.summary()}), flush=True)
            return None
        if args.path == "lookup":
            line = run_lookup(args, p, args.batch or 1024, torch, dev, R, ClockSampler)
        else:
            line = run_multi_lut(args, p, batch, torch, dev, R, ClockSampler)
        print(json.dumps(line), flush=True)
        return None

    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", init_method="env://")
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)

    import paper_2609_16915_gb300 as R
    from paper_2609_16915_gb300 import multi
    R.load()

    def d(a):
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int64)).to(dev)

    # workload: uniform-word keys (indistinguishable from real keys; the cost
    # does not depend on key values) and uniform ciphertexts, all resident
    bsk, ksk = W.uniform_keys(p)
    lwe = d(W.uniform_ciphertexts(p, batch, sub=rank))
    lut = d(W.lut_torus(p))
    out = torch.empty((batch, p.n + 1), dtype=torch.int64, device=dev)
    big = torch.empty((batch, p.kN + 1), dtype=torch.int64, device=dev)
    ctx = R.Context(p, device=local, max_batch=batch)
    ctx.upload_bsk(d(bsk))
    ctx.upload_ksk(d(ksk))
    del bsk, ksk
    stream = torch.cuda.current_stream(dev)
    ctx.sync_status(stream)
    flush = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.int32, device=dev)  # 256 MB > L2

    def barrier():
        if dist:
            dist.barrier()
        torch.cuda.synchronize(dev)

    for _ in range(max(3, args.warmup)):
        ctx.pbs_batch(lwe, lut, out, stream)
    ctx.sync_status(stream)

    # timed region: K steps, each bracketed by events; L2 flushed between steps
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    barrier()
    with ClockSampler(local) as clk:
        wall0 = time.perf_counter()
        for s in range(args.steps):
            flush.zero_()
            ev[s][0].record(stream)
            ctx.pbs_batch(lwe, lut, out, stream)
            ev[s][1].record(stream)
        barrier()
        wall = time.perf_counter() - wall0
    ctx.sync_status(stream)
    step_ms = [a.elapsed_time(b) for a, b in ev]
    total_ms = sum(step_ms)
    total_ms = multi.max_over_ranks(total_ms, dist, dev)
    value = world * batch * args.steps / (total_ms / 1e3)

    # dominant kernel (blind rotation) alone, same launch, events on its stream
    br_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(3)]
    ks_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(3)]
    for i in range(3):
        flush.zero_()
        br_ev[i][0].record(stream)
        ctx.blind_rotate_extract_batch(lwe, lut, big, stream)
        br_ev[i][1].record(stream)
        flush.zero_()
        ks_ev[i][0].record(stream)
        ctx.keyswitch_batch(big, out, stream)
        ks_ev[i][1].record(stream)
    ctx.sync_status(stream)
    br_ms = statistics.mean(a.elapsed_time(b) for a, b in br_ev)
    ks_ms = statistics.mean(a.elapsed_time(b) for a, b in ks_ev)

    # end to end through the public API with pinned host buffers
    h_in = torch.from_numpy(W.uniform_ciphertexts(p, batch, sub=rank).view(np.int64)).pin_memory()
    h_out = torch.empty((batch, p.n + 1), dtype=torch.int64).pin_memory()
    h_lut = torch.from_numpy(W.lut_torus(p).view(np.int64)).pin_memory()
    ctx.pbs_batch(h_in, h_lut, h_out, stream)
    barrier()
    e2e_steps = max(1, min(args.steps, 5))
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        ctx.pbs_batch(h_in, h_lut, h_out, stream)   # copies in, PBS, copies out, synchronises
    e2e_s = (time.perf_counter() - t0) / e2e_steps
    e2e_value = world * batch / multi.max_over_ranks(e2e_s, dist, dev)

    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    pk = peaks()
    sm_max = pk.get("sm_max_mhz", 2070.0)
    alu_peak = sms * 128 * sm_max * 1e6 / 1e12   # T int32 ops/s: SMs x 128 lanes x max clock
    br_ops, ks_ops = int_ops_per_pbs(p)
    achieved = br_ops * batch / (br_ms / 1e3) / 1e12
    # the same count against the measured rate of the NTT butterfly (three
    # multiplies, one of them a high product, and two adds: the integer
    # multiply pipe bounds it below the 128-lane issue limit): every counted
    # operation at the rate the butterfly's 8 counted operations run
    rates = measure_int_rates(torch, dev)
    primes = ctx.ntt_primes()
    bfly_per_clk = butterfly_rate(rates, primes)
    mix_peak = bfly_per_clk * 8 * sms * sm_max * 1e6 / 1e12
    pbs_roof = alu_peak * 1e12 / (br_ops + ks_ops)
    limbs = ks_tensor_limbs(p, batch)
    if limbs:
        ks_tf = ks_tensor_flops(p, batch, limbs) / (ks_ms / 1e3) / 1e12
        bf16_peak = pk.get("bf16_tflops", 1900.0)
        ks_roof = {"bound": "tensor", "kernel": "ks_digits_kernel + ks_tc_kernel (bf16 tcgen05)",
                   "achieved": ks_tf, "peak": bf16_peak, "unit": "TFLOP/s", "frac": ks_tf / bf16_peak,
                   "limbs": limbs, "peak_basis": "bf16_tflops of MEASURED_PEAKS.json (burst)"}
    else:
        ks_roof = {"bound": "alu", "kernel": "keyswitch_kernel", "achieved": ks_ops * batch / (ks_ms / 1e3) / 1e12,
                   "peak": alu_peak, "unit": "Tops/s (int32)"}
        ks_roof["frac"] = ks_roof["achieved"] / alu_peak

    if rank != 0:
        if dist:
            dist.destroy_process_group()
        return
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": max(3, args.warmup), "ms_per_step": total_ms / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "u64", "data": "synthetic",
        "config": {"workload": describe(p, batch), "batch": batch, "parallelism": f"dp{world}" if world > 1 else "none",
                   "l2": "flushed between steps (256 MB write)", "keys": "uniform words, resident"},
        "roofline": {"bound": "alu", "kernel": kernel_name(primes), "achieved": achieved, "peak": alu_peak,
                     "unit": "Tops/s (int32)", "frac": achieved / alu_peak, "traffic": measured_traffic(p, batch),
                     "peak_basis": f"{sms} SMs x 128 int32 lanes x {sm_max:.0f} MHz (sm_max_mhz of MEASURED_PEAKS.json)",
                     "kernel_ms": br_ms, "keyswitch_ms": ks_ms, "keyswitch": ks_roof,
                     "pbs_roof": pbs_roof, "pbs_frac_of_roof": value / world / pbs_roof,
                     "butterfly_rate_peak": mix_peak, "frac_of_butterfly_rate_peak": achieved / mix_peak,
                     "butterflies_per_clk_per_sm": round(bfly_per_clk, 2),
                     "int_rates_per_clk_per_sm": {k: round(v["per_clk_per_sm"], 2) for k, v in rates.items()
                                                  if isinstance(v, dict)}},
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": batch * (p.n + 1) * 8 + lut.numel() * 8,
                "d2h_bytes_per_step": batch * (p.n + 1) * 8},
        "gpu_launches": (3 if limbs else 2) * args.steps,
        "clocks": clk.summary(),
        "wall_s_timed": wall,
    }
    if world == 1 and not args.no_other and args.config == "standard" and not args.batch:
        # the other rows, measured in the same run after the headline's timed
        # region (short runs: their own warm-up and steps, L2 flushed between
        # steps); uniform-word keys as above
        other = {}
        for name, st, wu in (("gpt2_mlp", 3, 2), ("llama_silu", 2, 1)):
            other[name] = measure_other_config(name, torch, dev, R, st, wu, sms, sm_max, rates)
        ml = run_multi_lut(_Steps(2, 1), p, batch, torch, dev, R, _NoClock)
        other["multi_lut"] = {k: ml[k] for k in ("metric", "value", "unit", "ms_per_step", "steps")}
        other["multi_lut"]["workload"] = ml["config"]["workload"]
        lk = run_lookup(_Steps(2, 1), p, 1024, torch, dev, R, _NoClock)
        other["lookup"] = {k: lk[k] for k in ("metric", "value", "unit", "ms_per_step", "steps")}
        other["lookup"]["workload"] = lk["config"]["workload"]
        other["lookup"]["blind_rotation_frac"] = lk["roofline"]["frac"]
        line["other_workloads"] = other
    if not args.no_cpu_baseline:
        import oracle as O
        O.build()
        cores = O.default_threads()
        sample = args.cpu_sample or 3 * cores  # three ciphertexts per core: about 13 s on 16 Grace cores
        r, dt, t = oracle_pbs_rate(p, sample, threads=cores)
        line["cpu_baseline"] = {"value": r, "unit": UNIT, "cores": t, "kind": "oracle",
                                "sample": f"{sample} ciphertexts of the workload, uniform-word keys, {dt:.1f} s"}
    print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
