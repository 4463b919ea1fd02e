#!/usr/bin/env python
"""Benchmark of the masked MoE layer forward with its expert cache on GB300 (one JSON line).

Workload (default): a Mixtral-8x7B-shaped MoE layer decoding (d = 4096, E = 8, K = 2, SwiGLU width
14336, bf16) at batch 16 over a 512-step AR(1) hidden-state stream (rho = 0.8), routed with the soft
prior of a random keep-4-of-8 mask (pi = softmax(2 m)), with a 4-slot LRU expert cache whose misses
are fetched from pinned host memory. One step = routing + cache decision + fetch of missed experts
+ expert FFN + combine for one decode position of all 16 rows. Also reported: the same at batch 1,
and the masked fine-tuning / prefill forward (T = 4096 tokens, hard mask keeping 4 of 8 experts).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl mcft|reference]

Under torchrun (N > 1) every rank runs an independent replica on its own GPU (weak scaling; the
forward has no exchange step); rank 0 prints the line.
"""
from __future__ import annotations

import os

_CORES = os.cpu_count() or 1
for _v in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
    os.environ.setdefault(_v, str(_CORES))

import argparse  # noqa: E402
import json  # noqa: E402
import statistics  # noqa: E402
import subprocess  # noqa: E402
import sys  # noqa: E402
import threading  # noqa: E402
import time  # noqa: E402

import numpy as np  # noqa: E402
import torch  # noqa: E402

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2609_34077_gb300 import inputs as I  # noqa: E402

STREAM_STEPS = 512
METRIC = "masked MoE layer tokens/s"

# DRAM traffic per launch / algorithmic bytes, from one ncu capture of the kernel, keyed by the
# first 16 hex digits of the kernel source's sha256: when the source has changed since the
# capture, the bench reports traffic as null.
TRAFFIC = {
    "ffn13_decode": ("paper_2609_34077_gb300/csrc/ffn_decode.cu", "393328975a2ceb3d", None),
    "ffn2_decode": ("paper_2609_34077_gb300/csrc/ffn_decode.cu", "393328975a2ceb3d", None),
    "ffn_decode": ("paper_2609_34077_gb300/csrc/ffn_decode.cu", "393328975a2ceb3d", 1.0016),
    # DRAM traffic / (weights of the step's experts read once + activations + fetched bytes written)
    "ffn_decode_fetch": ("paper_2609_34077_gb300/csrc/ffn_decode.cu", "393328975a2ceb3d", 0.898),
    "fetch": ("paper_2609_34077_gb300/csrc/cache.cu", "68e0415de46353e9", 0.9253),
}


def traffic_ratio(kernel):
    import hashlib

    if kernel not in TRAFFIC:
        return None
    src, digest, ratio = TRAFFIC[kernel]
    cur = hashlib.sha256(open(os.path.join(ROOT, src), "rb").read()).hexdigest()[:16]
    if cur != digest:
        print(f"bench: {src} changed since the ncu capture of {kernel} "
              f"(sha {cur}, captured {digest}): traffic for {kernel} reported as null",
              file=sys.stderr)
        return None
    return ratio


# ------------------------------------------------------------------------------------------------
# host-side helpers (also exercised by the CPU multi-process tests)

def dist_env():
    return int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)), \
        int(os.environ.get("LOCAL_RANK", 0))


def replica_seed(base: int, rank: int) -> int:
    """Each replica decodes its own streams (weak scaling)."""
    return base + 1000 * rank


def aggregate(elapsed_s: float, units: float, world: int, group=None):
    """Max elapsed over ranks and summed units (tokens) -> (max_elapsed, total_units)."""
    if world == 1:
        return elapsed_s, units
    import torch.distributed as dist

    t = torch.tensor([elapsed_s], dtype=torch.float64)
    u = torch.tensor([units], dtype=torch.float64)
    if dist.get_backend(group) == "nccl":
        t, u = t.cuda(), u.cuda()
    dist.all_reduce(t, op=dist.ReduceOp.MAX, group=group)
    dist.all_reduce(u, op=dist.ReduceOp.SUM, group=group)
    return float(t.item()), float(u.item())


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return dict(hbm=d["hbm_gbs"], bf16=d["bf16_tflops"], bf16_sust=d.get("bf16_tflops_sustained"),
                    src="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sust=1700.0, src="fallback")


class ClockSampler:
    """nvidia-smi samples (SM clock, max, throttle reasons) during the timed region."""
    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index, self.lines, self.proc = index, [], None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.th = threading.Thread(target=self._read, daemon=True)
            self.th.start()
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *a):
        time.sleep(0.25)
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
            f = [v.strip() for v in ln.split(",")]
            if len(f) < 8:
                continue
            try:
                sm.append(float(f[0]))
                mx = float(f[1])
            except ValueError:
                continue
            for n, v in zip(names, f[4:8]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


# ------------------------------------------------------------------------------------------------

class DecodeLayer:
    """One MoE layer in decode: router + pinned host expert pool + device cache + workspace."""

    def __init__(self, shape, batch, seed, dev):
        from paper_2609_34077_gb300 import mcft as M

        self.M, self.shape, self.batch, self.dev = M, shape, batch, dev
        self.desc = M.desc_of(shape)
        self.lw = I.layer_weights(seed, shape, pin=True)
        self.prior = I.prior_from_mask(I.keep_mask(seed, shape.E, shape.keep))
        self.x_host = I.ar1_streams(seed, shape, STREAM_STEPS, batch).pin_memory()
        self.x = self.x_host.to(dev)
        self.wr = self.lw.router.to(dev)
        self.shared = [b.to(dev) for b in self.lw.shared]
        self.cache = None
        self.new_cache()
        self.ws = torch.empty(M.mcft_moe_workspace_size(self.desc, batch), dtype=torch.uint8, device=dev)
        self.idx = torch.empty((STREAM_STEPS, batch, shape.K), dtype=torch.int32, device=dev)
        self.gate = torch.empty((STREAM_STEPS, batch, shape.K), dtype=torch.float32, device=dev)
        self.y = torch.empty((batch, shape.d), dtype=torch.bfloat16, device=dev)
        self.compute = torch.cuda.current_stream(dev)
        self.copy = torch.cuda.Stream(dev)

    def new_cache(self):
        """Replace the expert cache by an empty one (same slots, policy and host pool)."""
        torch.cuda.synchronize(self.dev)
        if self.cache is not None:
            self.M.mcft_cache_destroy(self.cache)
        self.cache = self.M.mcft_cache_create(1, self.shape.E, self.shape.cache_slots,
                                              self.shape.expert_bytes, self.lw.experts,
                                              max_assign=self.batch * self.shape.K)

    def step(self, s, x=None, path="device"):
        """One decode step. path "device": the cache step's kernel publishes the expert table and
        a kernel fetches the misses while the hit experts are computed (no host round trip);
        path "host": the host reads the miss list, issues one copy per miss on the copy stream,
        then launches the forward."""
        M, p = self.M, s % STREAM_STEPS
        x = self.x[p] if x is None else x
        M.mcft_route(self.desc, x, self.wr, M.MCFT_ROUTE_SOFT_PRIOR, prior=self.prior,
                     idx=self.idx[p], gate=self.gate[p], stream=self.compute)
        M.mcft_cache_step(self.cache, 0, self.idx[p], stream=self.compute)
        if path == "device":
            M.mcft_moe_forward_cached(self.desc, x, self.idx[p], self.gate[p], self.cache, 0,
                                      self.shared, y=self.y, workspace=self.ws,
                                      compute_stream=self.compute, copy_stream=self.copy)
        else:
            ptrs = M.mcft_fetch_experts(self.cache, 0, self.compute, self.copy)
            M.mcft_moe_forward(self.desc, x, self.idx[p], self.gate[p], ptrs, self.shared, y=self.y,
                               workspace=self.ws, stream=self.compute)
        return self.y


def time_steps(fn, first, steps, stream):
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for s in range(first, first + steps):
        fn(s)
    b.record(stream)
    torch.cuda.synchronize()
    return a.elapsed_time(b) / 1e3


def host_link_probe(dev, nbytes):
    """Pinned host -> device bandwidth (GB/s) of nbytes by two methods: the copy engines (one
    copy, and the same bytes split into 2 and 4 concurrent copies on separate streams) and SM
    loads (the fetch kernel's copy loop, mcft_host_copy, on 38 / 76 / 152 CTAs); best of 10 (one
    copy) or 5 (the others). Returns the rates and their best."""
    from paper_2609_34077_gb300 import mcft as M

    src = torch.empty(nbytes, dtype=torch.uint8).pin_memory()
    dst = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    cur = torch.cuda.current_stream(dev)
    res = {}

    def best_of(reps, enqueue):
        best = 0.0
        for _ in range(reps):
            torch.cuda.synchronize()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(cur)
            enqueue(a)
            b.record(cur)
            torch.cuda.synchronize()
            best = max(best, nbytes / (a.elapsed_time(b) / 1e3) / 1e9)
        return best

    for n in (1, 2, 4):
        streams = [torch.cuda.Stream(dev) for _ in range(n)]
        chunk = -(-nbytes // n)

        def copies(start, streams=streams, chunk=chunk):
            for i, st in enumerate(streams):
                st.wait_event(start)
                with torch.cuda.stream(st):
                    dst[i * chunk:(i + 1) * chunk].copy_(src[i * chunk:(i + 1) * chunk],
                                                         non_blocking=True)
            for st in streams:
                cur.wait_stream(st)

        res[f"copy_engine_{n}_streams_gbs"] = best_of(10 if n == 1 else 5, copies)
    for blocks in (38, 76, 152):
        res[f"sm_loads_{blocks}_ctas_gbs"] = best_of(
            5, lambda start, blocks=blocks: M.mcft_host_copy(dst, src, blocks, stream=cur))
    M.mcft_device_error()
    res["best_gbs"] = max(res.values())
    del src, dst
    return res


def unique_per_step(idx_steps):
    return [len(torch.unique(i)) for i in idx_steps]


def decode_alg_bytes(U, steps, batch, shape):
    """Algorithmic DRAM bytes of the decode FFN over `steps` steps (U: distinct routed experts of
    each step): the W1 and W3 rows (GEMM13) and the W2 rows (GEMM2) of every expert the step
    computes (its routed experts and the shared experts, which every token uses), read once, plus
    the token activations in and out. Returns (GEMM13 bytes, GEMM2 bytes)."""
    S = shape.n_shared
    sel = sum(U) + steps * S
    T, K, d, w = batch, shape.K, shape.d, shape.w
    rows = T * (K + S)  # permuted rows per step: one per routed assignment and per shared expert
    b13 = sel * 2 * w * d * 2 + steps * (T * d * 2 + rows * w * 2)
    b2 = sel * w * d * 2 + steps * rows * (w * 2 + d * 4)
    return b13, b2


def decode_roofline(prof, U, steps, batch, shape, peaks):
    """HBM roofline of the decode FFN kernels. Algorithmic bytes per launch: the W1 and W3 rows
    (GEMM13) or W2 rows (GEMM2) of every expert the step computes, read once (the routed experts
    it selected and the shared experts, which every token uses), plus the token activations in and
    out; the fused kernel (both GEMMs in one launch) reads all three. Returns (dominant kernel's
    roofline dict, {kernel: GB/s})."""
    b13, b2 = decode_alg_bytes(U, steps, batch, shape)
    alg = {"ffn13_decode": b13, "ffn2_decode": b2, "ffn_decode": b13 + b2}
    rates, best = {}, None
    for k, b in alg.items():
        n, ms = prof.get(k, (0, 0.0))
        if not ms:
            continue
        rates[k] = b / (ms / 1e3) / 1e9
        if best is None or ms > prof[best][1]:
            best = k
    if best is None:
        return None, rates
    n, ms = prof[best]
    per_launch = alg[best] / max(1, n)
    tr = traffic_ratio(best)
    roof = dict(bound="hbm", achieved=rates[best], peak=peaks["hbm"], unit="GB/s",
                frac=rates[best] / peaks["hbm"], traffic=tr * per_launch if tr else None,
                kernel=best, peak_source=peaks["src"] + " hbm_gbs", alg_bytes_per_launch=per_launch,
                launches=n)
    return roof, rates


# Launches that move experts over the host link in a device-driven step: the fetch kernel on the
# copy stream (batches of more than 16 tokens, or a prefetch in flight), or the decode FFN launch
# that fetches its own misses (smaller batches).
FETCHING = ("fetch", "ffn_decode_fetch")


def fetching_kernel(kernels):
    """Name of the launch that fetched the misses in a profiled device-driven pass."""
    for k in FETCHING:
        if kernels.get(k, {}).get("launches", 0):
            return k
    return None


def decode_pass(L, first, steps, path="device", profile=False, e2e=False, clocks=None, world=1,
                record=None):
    """One measured pass over the decode steps [first, first + steps) of layer L.

    The pass starts from an empty cache and runs the untimed steps 0 .. first - 1 first, so every
    pass makes the same cache decisions and moves the same bytes over the same steps. With
    `profile` the library brackets each kernel with CUDA events (per-kernel times; a pass of its
    own, so the instrumentation never touches the headline time). With `e2e` every step also copies
    its hidden states from pinned host memory to the device and its output back to pinned host
    memory, on the compute stream inside the timed region. Returns (elapsed seconds, (hits,
    fetches, bypass) over the timed steps, per-kernel profile or None, bytes copied per step).
    With `record` (a list; untimed passes only) each step is synchronised and its fetch count
    appended."""
    M = L.M
    L.new_cache()
    for s in range(first):
        L.step(s, path=path)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    c0 = M.mcft_cache_stats(L.cache, 0)
    io_bytes = (0, 0)
    if e2e:
        xd = torch.empty((L.batch, L.shape.d), dtype=torch.bfloat16, device=L.dev)
        y_host = torch.empty((L.batch, L.shape.d), dtype=torch.bfloat16).pin_memory()

        def fn(s):
            xd.copy_(L.x_host[s % STREAM_STEPS], non_blocking=True)
            y = L.step(s, x=xd, path=path)
            y_host.copy_(y, non_blocking=True)

        io_bytes = (xd.numel() * 2, y_host.numel() * 2)
    else:
        def fn(s):
            L.step(s, path=path)
    if record is not None:
        def fn(s, step=fn):
            before = M.mcft_cache_stats(L.cache, 0)[1]
            step(s)
            record.append(int(M.mcft_cache_stats(L.cache, 0)[1] - before))
    if profile:
        M.mcft_profile_reset()
        M.mcft_profile_enable(True)
    if clocks is not None:
        with clocks:
            elapsed = time_steps(fn, first, steps, L.compute)
    else:
        elapsed = time_steps(fn, first, steps, L.compute)
    prof = None
    if profile:
        M.mcft_profile_enable(False)
        prof = M.mcft_profile_read()
    if world > 1:
        torch.distributed.barrier()
    M.mcft_device_error()
    c1 = M.mcft_cache_stats(L.cache, 0)
    return elapsed, tuple(int(b - a) for a, b in zip(c0, c1)), prof, io_bytes


def step_floor(d, link_gbs, hbm_gbs):
    """Lower bounds of a device-driven decode step from its own byte counts: the host link moving
    the step's misses (the FFN of the hits and of streamed misses can run under it), and that plus
    the missed experts' FFN read at HBM speed after their bytes land; each no less than the step's
    FFN bytes at HBM speed. From per-step means (link_ms, ...), and, with `per_step` counts in d,
    as the mean over steps of each step's own bound (step_ms, ...: tighter, since a step without
    a miss still streams its FFN). Fractions are bound / measured step time."""
    ms = d["ms_per_step"]
    fb, ffn = d["fetch_bytes_per_step"], d["ffn_dram_bytes_per_step"]
    lk, hb = link_gbs * 1e6, hbm_gbs * 1e6  # bytes per ms
    link_ms = max(fb / lk, ffn / hb)
    both_ms = max(fb / lk + fb / hb, ffn / hb)
    out = dict(link_ms=link_ms, link_plus_miss_ffn_ms=both_ms, frac_of_link=link_ms / ms,
               frac_of_link_plus_miss_ffn=both_ms / ms, link_gbs=link_gbs, hbm_gbs=hbm_gbs)
    ps = d.get("per_step")
    if ps and ps["fetches"] and len(ps["fetches"]) == len(ps["ffn_bytes"]):
        eb = ps["expert_bytes"]
        one = [max(f * eb / lk, b / hb) for f, b in zip(ps["fetches"], ps["ffn_bytes"])]
        two = [max(f * eb / lk + f * eb / hb, b / hb) for f, b in zip(ps["fetches"], ps["ffn_bytes"])]
        out.update(step_ms=sum(one) / len(one), step_plus_miss_ffn_ms=sum(two) / len(two),
                   frac_of_step=sum(one) / len(one) / ms,
                   frac_of_step_plus_miss_ffn=sum(two) / len(two) / ms)
    return out


def run_decode(shape, batch, steps, warmup, seed, dev, peaks, clocks=None, world=1, e2e=False):
    """Decode `steps` timed steps of one layer after `warmup` untimed ones, in four measured passes
    over the same steps from the same cache state (decode_pass), after one untimed pass:
      1. the headline time: device-driven fetch, no instrumentation (clocks sampled here);
      2. with `e2e`: the same with host <-> device copies of each step's inputs and output;
      3. the same as 1 with per-kernel CUDA events (kernel times, launches, FFN and fetch rooflines);
      4. the host-driven fetch (host reads the miss list, copy engine), kernels timed: the expert
         FFN then runs alone on the GPU.
    Returns (result dict, GPU routing ids [512, batch, K] on the host, elapsed seconds of pass 1)."""
    L = DecodeLayer(shape, batch, seed, dev)
    # an untimed pass over the same steps first: the first reads of the pinned host pool map its
    # pages for the device, which later passes (and any long-running decode) no longer pay; it
    # records each step's fetches (every pass makes the same decisions)
    per_step_fetches = []
    decode_pass(L, warmup, steps, record=per_step_fetches)
    elapsed, cnt, _, _ = decode_pass(L, warmup, steps, clocks=clocks, world=world)
    passes = {"timed": cnt}
    e2e_res = None
    if e2e:
        el_e, cnt_e, _, (bi, bo) = decode_pass(L, warmup, steps, e2e=True)
        passes["e2e"] = cnt_e
        e2e_res = dict(value=batch * steps / el_e, elapsed_s=el_e, unit="tokens/s", h2d_bytes_per_step=bi,
                       d2h_bytes_per_step=bo, ms_per_step=el_e * 1e3 / steps,
                       steps="the same decode steps as value, from the same cache state")
    el_p, cnt_p, prof, _ = decode_pass(L, warmup, steps, profile=True)
    passes["profiled"] = cnt_p
    el_h, cnt_h, hprof, _ = decode_pass(L, warmup, steps, path="host", profile=True)
    passes["host_fetch"] = cnt_h
    pos = [s % STREAM_STEPS for s in range(warmup, warmup + steps)]
    U = unique_per_step([L.idx[p] for p in pos])
    hits, fetches, byp = cnt
    roof, rates = decode_roofline(prof, U, steps, batch, shape, peaks)
    roof_alone, rates_alone = decode_roofline(hprof, U, steps, batch, shape, peaks)
    fetch_bytes = fetches * shape.expert_bytes / steps
    b13, b2 = decode_alg_bytes(U, steps, batch, shape)
    out = dict(
        per_step=dict(fetches=per_step_fetches, experts=U, expert_bytes=shape.expert_bytes,
                      ffn_bytes=[sum(decode_alg_bytes([u], 1, batch, shape)) for u in U]),
        tokens_per_s=batch * steps / elapsed, ms_per_step=elapsed * 1e3 / steps, steps=steps,
        warmup=warmup, fetch_path="device", hits=hits, fetches=fetches, bypass=byp,
        fetches_per_step=fetches / steps, fetches_per_token=fetches / (steps * batch),
        hit_rate=hits / max(1, hits + fetches), mean_experts_per_step=float(np.mean(U)),
        fetch_bytes_per_step=fetch_bytes,
        passes_same_decisions=all(c == cnt for c in passes.values()),
        ffn_dram_bytes_per_step=(b13 + b2) / steps,
        profiled_ms_per_step=el_p * 1e3 / steps,
        kernels={k: dict(launches=v[0], ms=round(v[1], 4)) for k, v in prof.items() if v[0]},
        gpu_launches=int(sum(v[0] for v in prof.values() if v[0])), roofline=roof,
        kernel_gbs=rates,
        kernel_ms_per_step=sum(v[1] for k, v in prof.items() if k not in FETCHING) / steps,
        fetch_launch_ms_per_step=sum(v[1] for k, v in prof.items() if k in FETCHING) / steps,
        roofline_alone=dict(roof_alone or {}, note="same FFN kernel in the host-driven step, "
                            "where it runs alone"),
        host_fetch_path=dict(tokens_per_s=batch * steps / el_h, ms_per_step=el_h * 1e3 / steps,
                             kernel_gbs=rates_alone),
    )
    if e2e_res is not None:
        out["e2e"] = e2e_res
    idx_host = L.idx.cpu().numpy()
    del L
    torch.cuda.empty_cache()
    return out, idx_host, elapsed


class DecodeStack:
    """L MoE layers decoding at batch 1, each with its own router, soft prior (random keep-k
    mask), AR(1) hidden-state stream and B cache slots; layers are not chained. The pinned host
    pool holds E distinct expert blocks that every layer aliases (a 32-layer Mixtral pool would be
    90 GB): fetch counts and bytes are those of distinct per-layer experts.

    With the device-driven fetch a step has no host synchronisation, so `capture()` records one
    step of all L layers as a CUDA graph; `step()` then copies the token's hidden states into the
    graph's input buffer and replays it (one launch per token instead of ~10 per layer)."""

    def __init__(self, shape, L, steps, seed, dev, policy="LRU", path="device"):
        from paper_2609_34077_gb300 import mcft as M

        self.M, self.shape, self.L, self.dev, self.path = M, shape, L, dev, path
        self.desc = M.desc_of(shape)
        pool = I.layer_weights(seed, shape, layer=0, pin=True)
        self.pool = pool
        self.shared = [b.to(dev) for b in pool.shared]
        self.routers, self.priors = [], []
        x = torch.empty((steps, L, shape.d), dtype=torch.bfloat16)
        for l in range(L):
            self.routers.append(I.router_weight(seed, shape, l).to(dev))
            self.priors.append(I.prior_from_mask(I.keep_mask(seed, shape.E, shape.keep, l)))
            x[:, l] = I.ar1_streams(seed, shape, steps, 1, l)[:, 0]
        self.x = x.to(dev)                      # [steps, L, d]
        self.xin = torch.empty((L, shape.d), dtype=torch.bfloat16, device=dev)
        host = [pool.experts[e] for _ in range(L) for e in range(shape.E)]
        self.cache = M.mcft_cache_create(L, shape.E, shape.cache_slots, shape.expert_bytes, host,
                                         max_assign=shape.K, policy=policy)
        self.ws = torch.empty(M.mcft_moe_workspace_size(self.desc, 1), dtype=torch.uint8, device=dev)
        self.idx = torch.empty((L, shape.K), dtype=torch.int32, device=dev)
        self.gate = torch.empty((L, shape.K), dtype=torch.float32, device=dev)
        self.y = torch.empty((L, shape.d), dtype=torch.bfloat16, device=dev)
        self.compute = torch.cuda.Stream(dev)
        self.copy = torch.cuda.Stream(dev)
        self.graph = None

    def layers(self):
        """Enqueue one decode step of every layer on the compute stream (inputs in self.xin)."""
        M = self.M
        for l in range(self.L):
            x = self.xin[l:l + 1]
            M.mcft_route(self.desc, x, self.routers[l], M.MCFT_ROUTE_SOFT_PRIOR, prior=self.priors[l],
                         idx=self.idx[l:l + 1], gate=self.gate[l:l + 1], stream=self.compute)
            M.mcft_cache_step(self.cache, l, self.idx[l:l + 1], stream=self.compute)
            if self.path == "device":
                M.mcft_moe_forward_cached(self.desc, x, self.idx[l:l + 1], self.gate[l:l + 1],
                                          self.cache, l, self.shared, y=self.y[l:l + 1],
                                          workspace=self.ws, compute_stream=self.compute,
                                          copy_stream=self.copy)
            else:
                ptrs = M.mcft_fetch_experts(self.cache, l, self.compute, self.copy)
                M.mcft_moe_forward(self.desc, x, self.idx[l:l + 1], self.gate[l:l + 1], ptrs,
                                   self.shared, y=self.y[l:l + 1], workspace=self.ws,
                                   stream=self.compute)

    def capture(self):
        assert self.path == "device"
        self.graph = torch.cuda.CUDAGraph()
        torch.cuda.synchronize()
        with torch.cuda.graph(self.graph, stream=self.compute):
            self.layers()
        torch.cuda.synchronize()

    def step(self, s):
        # input copy, then the step, in order on the compute stream (replay() launches the graph
        # on the current stream)
        with torch.cuda.stream(self.compute):
            self.xin.copy_(self.x[s], non_blocking=True)
            if self.graph is not None:
                self.graph.replay()
            else:
                self.layers()


def run_stack(shape, L, steps, warmup, seed, dev, policy="LRU", path="device", graph=False):
    """Decode `warmup + steps` tokens through an L-layer stack; TPOT over the last `steps`.
    With graph=True the step is captured after the warm-up and replayed (no per-kernel timing)."""
    from paper_2609_34077_gb300 import mcft as M

    S = DecodeStack(shape, L, warmup + steps + 1, seed, dev, policy, path)
    for s in range(warmup):
        S.step(s)
    torch.cuda.synchronize()
    if graph:
        # the capture records the step but also runs nothing; the cache is untouched by it
        S.capture()
    h0, f0, b0 = M.mcft_cache_stats(S.cache, -1)
    M.mcft_profile_reset()
    M.mcft_profile_enable(not graph)
    elapsed = time_steps(S.step, warmup, steps, S.compute)
    M.mcft_profile_enable(False)
    prof = M.mcft_profile_read()
    M.mcft_device_error()
    h1, f1, b1 = M.mcft_cache_stats(S.cache, -1)
    hits, fetches = h1 - h0, f1 - f0
    res = dict(workload=f"{shape.name} decode stack, {L} layers, batch 1, {policy}",
               layers=L, policy=policy, fetch_path=path, cuda_graph=graph, steps=steps,
               warmup=warmup, tpot_ms=elapsed * 1e3 / steps, tokens_per_s=steps / elapsed,
               fetches_per_token=fetches / steps, hit_rate=hits / max(1, hits + fetches),
               fetches_per_token_whole_stream=f1 / (warmup + steps),
               hit_rate_whole_stream=h1 / max(1, h1 + f1),
               fetch_gb_per_token=fetches * shape.expert_bytes / steps / 1e9,
               link_bound_tpot_ms=fetches * shape.expert_bytes / steps / 210e9 * 1e3,
               host_pool="E distinct pinned blocks aliased by every layer")
    if not graph:
        res.update(kernel_ms_per_token=sum(v[1] for v in prof.values()) / steps,
                   gpu_launches=int(sum(v[0] for v in prof.values())),
                   kernels={k: dict(launches=v[0], ms=round(v[1], 3)) for k, v in prof.items() if v[0]})
    del S
    torch.cuda.empty_cache()
    return res


class ChainStack:
    """L chained MoE layers (mcft_stack: residual stream, per-layer RMSNorm, soft-prior routing,
    device cache with device-driven fetch, optional prefetch of each next layer's predicted
    experts) decoding at batch 1. Each layer has its own router, RMSNorm scale and random soft-prior
    mask; the pinned host pool holds E distinct expert blocks that every layer aliases (as in
    DecodeStack). The stream entering layer 0 is the AR(1) recipe in fp32, one row per token."""

    def __init__(self, shape, L, steps, seed, dev, policy="LRU", n_prefetch=0):
        from paper_2609_34077_gb300 import mcft as M

        self.M, self.shape, self.L, self.dev = M, shape, L, dev
        desc = M.desc_of(shape)
        pool = I.layer_weights(seed, shape, layer=0, pin=True)
        self.pool = pool
        shared = [b.to(dev) for b in pool.shared]
        routers = [I.router_weight(seed, shape, l).to(dev) for l in range(L)]
        gammas = [I.norm_weight(seed, shape, l).to(dev) for l in range(L)]
        priors = np.stack([I.prior_from_mask(I.keep_mask(seed, shape.E, shape.keep, l))
                           for l in range(L)])
        host = [pool.experts[e] for _ in range(L) for e in range(shape.E)]
        self.cache = M.mcft_cache_create(L, shape.E, shape.cache_slots, shape.expert_bytes, host,
                                         max_assign=shape.K, policy=policy)
        self.stack = M.mcft_stack_create(desc, routers, priors, gammas,
                                         [shared] * L if shape.n_shared else None, shape.norm_eps,
                                         self.cache, n_prefetch=n_prefetch, T_max=1)
        self.x0 = I.residual_stream(seed, shape, steps, 1).to(dev)  # [steps, 1, d]
        self.x = torch.empty((1, shape.d), dtype=torch.float32, device=dev)
        self.compute = torch.cuda.Stream(dev)
        self.copy = torch.cuda.Stream(dev)
        self.graph = None

    def capture(self):
        self.graph = torch.cuda.CUDAGraph()
        torch.cuda.synchronize()
        with torch.cuda.graph(self.graph, stream=self.compute):
            self.M.mcft_stack_step(self.stack, self.x, self.compute, self.copy)
        torch.cuda.synchronize()

    def step(self, s):
        with torch.cuda.stream(self.compute):
            self.x.copy_(self.x0[s], non_blocking=True)
            if self.graph is not None:
                self.graph.replay()
            else:
                self.M.mcft_stack_step(self.stack, self.x, self.compute, self.copy)


def run_chain(shape, L, steps, warmup, seed, dev, policy="LRU", n_prefetch=0, graph=True):
    """Decode `warmup + steps` tokens through a chained L-layer stack; TPOT over the last `steps`."""
    from paper_2609_34077_gb300 import mcft as M

    S = ChainStack(shape, L, warmup + steps + 1, seed, dev, policy, n_prefetch)
    torch.cuda.synchronize()
    for s in range(warmup):
        S.step(s)
    torch.cuda.synchronize()
    if graph:
        S.capture()  # records one step; runs nothing
    h0, f0, _ = M.mcft_cache_stats(S.cache, -1)
    p0, u0, m0 = M.mcft_cache_prefetch_stats(S.cache, -1)
    M.mcft_profile_reset()
    M.mcft_profile_enable(not graph)
    elapsed = time_steps(S.step, warmup, steps, S.compute)
    M.mcft_profile_enable(False)
    prof = M.mcft_profile_read()
    M.mcft_device_error()
    h1, f1, _ = M.mcft_cache_stats(S.cache, -1)
    p1, u1, m1 = M.mcft_cache_prefetch_stats(S.cache, -1)
    fetches, pref, useful = f1 - f0, p1 - p0, u1 - u0
    # bytes on the host link: every demand fetch in full, prefetches as far as they ran (a
    # prefetch the next step dropped stops early)
    moved = (fetches * shape.expert_bytes + (m1 - m0)) / steps
    res = dict(workload=f"{shape.name} chained decode stack, {L} layers, batch 1, {policy}, "
                        f"prefetch {n_prefetch or 'off'}",
               layers=L, policy=policy, n_prefetch=n_prefetch, cuda_graph=graph, steps=steps,
               warmup=warmup, tpot_ms=elapsed * 1e3 / steps, tokens_per_s=steps / elapsed,
               demand_fetches_per_token=fetches / steps, prefetches_per_token=pref / steps,
               useful_prefetches_per_token=useful / steps,
               prefetch_accuracy=useful / pref if pref else None,
               prefetch_gb_moved_per_token=(m1 - m0) / steps / 1e9,
               hit_rate=(h1 - h0) / max(1, h1 - h0 + fetches),
               link_gb_per_token=moved / 1e9, link_bound_tpot_ms=moved / 210e9 * 1e3,
               host_pool="E distinct pinned blocks aliased by every layer")
    if not graph:
        res.update(kernel_ms_per_token={k: round(v[1] / steps, 4) for k, v in prof.items() if v[0]},
                   launches_per_token={k: v[0] / steps for k, v in prof.items() if v[0]})
    del S
    torch.cuda.empty_cache()
    return res


def run_prefill(steps, warmup, seed, dev, peaks):
    from paper_2609_34077_gb300 import mcft as M

    sh, T = I.MIXTRAL, 4096
    desc = M.desc_of(sh)
    mask = I.keep_mask(seed, sh.E, 4)
    lw = I.layer_weights(seed, sh, experts=[int(e) for e in np.nonzero(mask)[0]])
    experts = [None if b is None else b.to(dev) for b in lw.experts]
    wr = lw.router.to(dev)
    x = I.hidden_iid(seed, sh, T).to(dev)
    ws = torch.empty(M.mcft_moe_workspace_size(desc, T), dtype=torch.uint8, device=dev)
    y = torch.empty_like(x)
    idx = torch.empty((T, sh.K), dtype=torch.int32, device=dev)
    gate = torch.empty((T, sh.K), dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)

    def step(s):
        M.mcft_route(desc, x, wr, M.MCFT_ROUTE_HARD_MASK, mask=mask, idx=idx, gate=gate, stream=stream)
        M.mcft_moe_forward(desc, x, idx, gate, experts, y=y, workspace=ws, stream=stream)

    for s in range(warmup):
        step(s)
    M.mcft_profile_reset()
    M.mcft_profile_enable(True)
    elapsed = time_steps(step, 0, steps, stream)
    M.mcft_profile_enable(False)
    prof = M.mcft_profile_read()
    M.mcft_device_error()
    A = T * sh.K
    f13 = 2.0 * A * sh.d * 2 * sh.w
    f2 = 2.0 * A * sh.w * sh.d
    n13, ms13 = prof["gemm13_tc"]
    n2, ms2 = prof["gemm2_tc"]
    peak = peaks["bf16"]
    res = dict(workload="mixtral-8x7b prefill T=4096 hard mask keep 4/8", tokens_per_s=T * steps / elapsed,
               ms_per_step=elapsed * 1e3 / steps, tflop_per_step=(f13 + f2) / 1e12,
               kernels={k: dict(launches=v[0], ms=round(v[1], 4)) for k, v in prof.items() if v[0]},
               gpu_launches=int(sum(v[0] for v in prof.values())))
    if ms13 and ms2:
        a13 = f13 / (ms13 / n13 / 1e3) / 1e12
        a2 = f2 / (ms2 / n2 / 1e3) / 1e12
        res["roofline"] = dict(bound="tensor", kernel="gemm13_tc", achieved=a13, peak=peak,
                               unit="TFLOP/s", frac=a13 / peak, flop_per_launch=f13)
        res["gemm2_tflops"] = a2
        res["gemm_frac_of_peak"] = (f13 + f2) / ((ms13 / n13 + ms2 / n2) / 1e3) / 1e12 / peak
    # the same steps on CTA-pair tiles (mcft_set_tc_tiles), for comparison with the default tiles
    M.mcft_set_tc_tiles(M.MCFT_TC_TILES_CTA_PAIR)
    try:
        ws = torch.empty(M.mcft_moe_workspace_size(desc, T), dtype=torch.uint8, device=dev)
        for s in range(warmup):
            step(s)
        M.mcft_profile_reset()
        M.mcft_profile_enable(True)
        el_p = time_steps(step, 0, steps, stream)
        M.mcft_profile_enable(False)
        pp = M.mcft_profile_read()
        M.mcft_device_error()
    finally:
        M.mcft_profile_enable(False)
        M.mcft_set_tc_tiles(M.MCFT_TC_TILES_ONE_CTA)
    (p13, t13), (p2, t2) = pp["gemm13_tc_pair"], pp["gemm2_tc_pair"]
    if t13 and t2:
        res["cta_pair_tiles"] = dict(
            note="same steps with mcft_set_tc_tiles(CTA_PAIR): 256 x 256 tiles on 2-CTA clusters",
            ms_per_step=el_p * 1e3 / steps, gemm13_us=t13 / p13 * 1e3, gemm2_us=t2 / p2 * 1e3,
            gemm13_frac=f13 / (t13 / p13 / 1e3) / 1e12 / peak,
            gemm2_frac=f2 / (t2 / p2 / 1e3) / 1e12 / peak)
    return res


def _flush_l2(buf):
    buf.add_(1)  # writes 256 MB, twice the L2, so the next kernel starts from a cold L2


def time_calls(fn, n, stream, flush=None):
    """Mean device time (ms) of fn() over n calls, each bracketed by its own CUDA events on
    `stream`; with `flush` given, the L2 is flushed before every call (outside the events)."""
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(n)]
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        for a, b in evs:
            if flush is not None:
                _flush_l2(flush)
            a.record(stream)
            fn()
            b.record(stream)
    torch.cuda.synchronize()
    return sum(a.elapsed_time(b) for a, b in evs) / n


def run_read_probe(dev, peaks, reps=5):
    """One launch of the decode FFN's grid reading the decode FFN's weight bytes with no
    computation (mcft_read_probe): as one contiguous stream and with the FFN's own load pattern,
    the L2 flushed before each call, for the expert bytes of DeepSeek-shaped batch 1 (8 experts,
    138.4 MB) and Mixtral-shaped batch 1 / 16 (2 / 8 experts). What a launch of that shape reads
    at all, beside the FFN's roofline against the copy peak."""
    from paper_2609_34077_gb300 import mcft as M

    flush = torch.zeros(64 << 20, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)
    blocks = 2 * torch.cuda.get_device_properties(dev).multi_processor_count
    sink = torch.zeros(1, dtype=torch.int32, device=dev)
    out = {}
    for name, sh, n_exp in (("dsv2_b1", I.DSV2_LITE, 8), ("mixtral_b1", I.MIXTRAL, 2),
                            ("mixtral_b16", I.MIXTRAL, 8)):
        nbytes = n_exp * sh.expert_bytes
        buf = torch.empty(nbytes // 2, dtype=torch.bfloat16, device=dev)
        res = dict(bytes=nbytes, row_bytes=sh.d * 2, blocks=blocks)
        for pattern, key in ((0, "contiguous"), (1, "ffn_pattern")):
            f = lambda: M.mcft_read_probe(buf, pattern, row_bytes=sh.d * 2, blocks=blocks, sink=sink,
                                          stream=stream)
            f()
            ms = time_calls(f, reps, stream, flush=flush)
            gbs = nbytes / (ms / 1e3) / 1e9
            res[key] = dict(us=ms * 1e3, gbs=gbs, frac_of_copy_peak=gbs / peaks["hbm"])
        M.mcft_device_error()
        out[name] = res
        del buf
    del flush
    torch.cuda.empty_cache()
    return out


_BATCHES = {}


def _masked_batch(sh, T, seed, dev):
    """A fine-tuning batch under a hard mask keeping 75 % of the experts (compact ratio r = 75 %):
    the mask, the kept experts' weights (others absent), x and the hard-mask routing. Built once
    per shape and kept in _BATCHES for the LoRA and mask measurements (cleared by the caller)."""
    key = (sh.name, T, seed, str(dev))
    if key not in _BATCHES:
        _BATCHES[key] = _make_masked_batch(sh, T, seed, dev)
    return _BATCHES[key]


def _make_masked_batch(sh, T, seed, dev):
    from paper_2609_34077_gb300 import mcft as M

    mask = I.keep_mask(seed, sh.E, sh.E * 3 // 4)
    kept = [int(e) for e in np.nonzero(mask)[0]]
    lw = I.layer_weights(seed, sh, experts=kept)
    experts = [None if b is None else b.to(dev) for b in lw.experts]
    shared = [b.to(dev) for b in lw.shared]
    x = I.hidden_iid(seed, sh, T).to(dev)
    desc = M.desc_of(sh)
    idx, gate = M.mcft_route(desc, x, lw.router.to(dev), M.MCFT_ROUTE_HARD_MASK, mask=mask)
    return desc, kept, experts, shared, x, idx, gate


def lora_work(shape, T, rank):
    """Algorithmic work of a Stage-2 forward of T tokens, every permuted row adapted (rank r):
    bytes of the two tcgen05 down projections (each gathered x row and each h row read once,
    s [A1 x | A3 x] and s A2 h written in bf16) and FLOP of the base GEMMs, of the adapters' up
    projections (the extra k-blocks) and of their down projections."""
    rows = T * (shape.K + shape.n_shared)
    r, d, w = rank, shape.d, shape.w
    return dict(rows=rows,
                down_bytes=rows * (d * 2 + 2 * r * 2) + rows * (w * 2 + r * 2),
                base_flop=2.0 * rows * 3 * d * w,
                up_flop=2.0 * rows * (2 * w + d) * r,
                down_flop=2.0 * rows * (2 * d + w) * r)


def run_lora(steps, warmup, seed, dev, peaks, rank=8, shapes=(I.MIXTRAL, I.DSV2_LITE), T=4096):
    """The Stage-2 forward (experts of the fixed concentration set with rank-8 LoRA adapters,
    alpha 16; the shared experts adapted too) against the plain forward on the same batch: T tokens
    routed under a hard mask keeping 75 % of the experts. Both arms are timed in alternating
    blocks with CUDA events, then one profiled pass of the LoRA arm gives its kernels' times."""
    from paper_2609_34077_gb300 import mcft as M

    out = {}
    stream = torch.cuda.current_stream(dev)
    for sh in shapes:
        desc, kept, experts, shared, x, idx, gate = _masked_batch(sh, T, seed, dev)
        ad = [I.lora_block(seed, sh, e, rank).to(dev) if e in kept else None for e in range(sh.E)]
        sad = [I.lora_block(seed, sh, ("shared", s), rank).to(dev) for s in range(sh.n_shared)]
        ws = torch.empty(M.mcft_moe_workspace_size_lora(desc, rank, T), dtype=torch.uint8,
                         device=dev)
        y = torch.empty_like(x)
        scale = 16.0 / rank

        def plain(s):
            M.mcft_moe_forward(desc, x, idx, gate, experts, shared, y=y, workspace=ws, stream=stream)

        def lora(s):
            M.mcft_moe_forward_lora(desc, x, idx, gate, experts, shared, ad, sad, rank, scale, y=y,
                                    workspace=ws, stream=stream)

        for s in range(warmup):
            plain(s)
            lora(s)
        t_plain = t_lora = 0.0
        blocks = 4
        per = max(1, steps // blocks)
        for _ in range(blocks):
            t_plain += time_steps(plain, 0, per, stream)
            t_lora += time_steps(lora, 0, per, stream)
        n = blocks * per
        profs = []
        for fn in (plain, lora):
            M.mcft_profile_reset()
            M.mcft_profile_enable(True)
            time_steps(fn, 0, n, stream)
            M.mcft_profile_enable(False)
            profs.append(M.mcft_profile_read())
        prof_plain, prof = profs
        M.mcft_device_error()
        wk = lora_work(sh, T, rank)
        r = rank
        ld_bytes, f_base, f_up, f_down = (wk["down_bytes"], wk["base_flop"], wk["up_flop"],
                                          wk["down_flop"])
        nl, msl = prof.get("lora_down", (0, 0.0))
        n13, ms13 = prof.get("gemm13_tc", (0, 0.0))
        n2, ms2 = prof.get("gemm2_tc", (0, 0.0))
        res = dict(workload=f"{sh.name} T={T} hard mask keep {len(kept)}/{sh.E}, rank {r} "
                            f"adapters on the {len(kept)} kept and {sh.n_shared} shared experts",
                   tokens_per_s=T * n / t_lora, tokens_per_s_plain=T * n / t_plain,
                   ms_per_step=t_lora * 1e3 / n, ms_per_step_plain=t_plain * 1e3 / n,
                   lora_overhead=t_lora / t_plain - 1.0,
                   kernels={k: dict(launches=v[0], ms_per_step=round(v[1] / n, 4))
                            for k, v in prof.items() if v[0]},
                   kernels_plain={k: dict(launches=v[0], ms_per_step=round(v[1] / n, 4))
                                  for k, v in prof_plain.items() if v[0]},
                   gpu_launches_per_step=sum(v[0] for v in prof.values()) / n)
        if nl and msl:
            a = ld_bytes / (msl / n / 1e3) / 1e9
            res["roofline_lora_down"] = dict(
                bound="hbm", kernel="lora_down", achieved=a, peak=peaks["hbm"], unit="GB/s",
                frac=a / peaks["hbm"], alg_bytes_per_step=ld_bytes, launches_per_step=nl / n,
                note="x and h rows read once + bf16 U13 / U2 written; the adapters' A "
                     "matrices are L2-resident")
        if n13 and n2 and ms13 and ms2:
            a = (f_base + f_up) / ((ms13 + ms2) / n / 1e3) / 1e12
            res["roofline_gemm"] = dict(bound="tensor", kernel="gemm13_tc+gemm2_tc", achieved=a,
                                        peak=peaks["bf16"], unit="TFLOP/s", frac=a / peaks["bf16"],
                                        flop_per_step=f_base + f_up,
                                        note="base GEMM flops + the adapters' up projections "
                                             "(one extra k-block per adapted tile)")
        res["adapter_flop_share"] = (f_up + f_down) / (f_base + f_up + f_down)
        out[sh.name] = res
        del ad, sad, ws, y
        torch.cuda.empty_cache()
    return out


def gate_grad_bytes(shape, T):
    """Algorithmic bytes of one gate-gradient call: each routed row's fp32 expert output read
    once, dL/dy read once per token (bf16), the permuted row index read and dL/dg written."""
    rows = T * shape.K
    return rows * shape.d * 4 + T * shape.d * 2 + rows * 4 * 2


def run_mask(calls, warmup, seed, dev, peaks, T=4096):
    """The Stage-1 mask machinery on a fine-tuning batch of T tokens per shape, each kernel timed
    alone with the L2 flushed before every call: mcft_mask_sample for every layer at once
    (compact ratio 75 %), mcft_gate_grad after the layer forward (HBM: the forward's fp32 expert
    output rows and dL/dy), mcft_mask_grad for one layer (two small launches)."""
    from paper_2609_34077_gb300 import mcft as M

    out = {}
    stream = torch.cuda.current_stream(dev)
    flush = torch.zeros(64 << 20, dtype=torch.float32, device=dev)
    for sh, L in ((I.MIXTRAL, 32), (I.DSV2_LITE, 26)):
        desc, kept, experts, shared, x, idx, gate = _masked_batch(sh, T, seed, dev)
        keep = len(kept)
        g = np.random.default_rng(seed)
        m_t = torch.from_numpy(g.standard_normal((L, sh.E)).astype(np.float32)).to(dev)
        u = torch.from_numpy(I.uniforms(seed, (L, sh.E))).to(dev)
        mask, pi = M.mcft_mask_sample(m_t, u, keep, stream=stream)
        ws = torch.empty(M.mcft_moe_workspace_size(desc, T), dtype=torch.uint8, device=dev)
        y = torch.empty_like(x)
        M.mcft_moe_forward(desc, x, idx, gate, experts, shared, y=y, workspace=ws, stream=stream)
        dy = I.hidden_iid(seed + 1, sh, T, tag="dy").to(dev)
        dg = torch.empty((T, sh.K), dtype=torch.float32, device=dev)
        dm = torch.empty(sh.E, dtype=torch.float32, device=dev)
        dmt = torch.zeros(sh.E, dtype=torch.float32, device=dev)
        fns = dict(
            mask_sample=lambda: M.mcft_mask_sample(m_t, u, keep, stream=stream),
            gate_grad=lambda: M.mcft_gate_grad(desc, dy, ws, dgate=dg, stream=stream),
            mask_grad=lambda: M.mcft_mask_grad(desc, idx, gate, dg, pi[0], dm=dm, dm_tilde=dmt,
                                               accumulate=True, stream=stream))
        for f in fns.values():
            for _ in range(warmup):
                f()
        us = {k: 1e3 * time_calls(f, calls, stream, flush) for k, f in fns.items()}
        M.mcft_device_error()
        gg_bytes = gate_grad_bytes(sh, T)
        a = gg_bytes / (us["gate_grad"] / 1e6) / 1e9
        out[sh.name] = dict(
            workload=f"{sh.name} T={T}, {L} layers x {sh.E} experts, keep {keep}",
            us_per_call={k: round(v, 2) for k, v in us.items()},
            roofline_gate_grad=dict(bound="hbm", kernel="gate_grad", achieved=a, peak=peaks["hbm"],
                                    unit="GB/s", frac=a / peaks["hbm"], alg_bytes=gg_bytes,
                                    note="each routed row's fp32 expert output and its token's "
                                         "dL/dy read once; L2 flushed before each call"),
            mask_sample_note="one 32-thread block per layer: latency-bound, "
                             f"{L * sh.E * (4 + 4 + 1 + 4)} bytes in total (m~, u in; mask, pi out)")
        del ws, y, dy
        torch.cuda.empty_cache()
    del flush
    return out


# ------------------------------------------------------------------------------------------------
# CPU oracle timing (the reported baseline, and the reference arm)

def oracle_decode_tokens_per_s(shape, batch, seed, budget_s=12.0, lw=None, warmup=0, max_steps=None):
    """The CPU oracle (routing + LRU accounting + fp64 SwiGLU combine) on decode steps of the same
    stream: `warmup` untimed steps, then timed steps until `max_steps` or ~budget_s of work;
    returns (tokens/s, timed steps)."""
    import oracle

    lw = lw or I.layer_weights(seed, shape)
    prior = I.prior_from_mask(I.keep_mask(seed, shape.E, shape.keep))
    xs = I.ar1_streams(seed, shape, STREAM_STEPS, batch)
    wr = lw.router.double().numpy()
    ex = [tuple(t.double().numpy() for t in I.split_expert(b, shape)) for b in lw.experts]
    sh = [tuple(t.double().numpy() for t in I.split_expert(b, shape)) for b in lw.shared]
    cache = oracle.cache.SlotCache(shape.E, shape.cache_slots, "LRU")

    def step(i):
        x = xs[i % STREAM_STEPS].double().numpy()
        r = oracle.routing.route(x, wr, shape.K, oracle.routing.MODE_SOFT_PRIOR, shape.gate, prior=prior)
        cache.step(r["idx"])
        oracle.ffn.moe_layer(x, r["idx"], r["gate"], ex, sh)

    for i in range(warmup):
        step(i)
    limit = max_steps if max_steps else STREAM_STEPS
    t0 = time.perf_counter()
    n = 0
    while True:
        step(warmup + n)
        n += 1
        el = time.perf_counter() - t0
        if el >= budget_s or n >= limit:
            return batch * n / el, n


def oracle_fetch_check(shape, batch, seed, idx_gpu, first, steps):
    """Checks a decode run's routing and fetch counts against the CPU oracle (the metric's
    "fetches/token exact"): the oracle routes every stream position the run used (fp64, Eq.
    inference with the run's prior), the GPU's ids are compared with it token by token, and two
    oracle caches (Section 4.1 LRU) replay steps 0 .. first + steps - 1, one on the oracle's ids and
    one on the GPU's. Returns the counts over the timed steps [first, first + steps): tokens routed,
    near ties (relative gap between the K-th and (K+1)-th score below 1e-4), tokens whose ids differ
    from the oracle's (inside / outside the near-tie band) and hits and fetches of both replays."""
    import oracle

    n = first + steps
    xs = I.ar1_streams(seed, shape, STREAM_STEPS, batch)
    wr = I.router_weight(seed, shape).double().numpy()
    prior = I.prior_from_mask(I.keep_mask(seed, shape.E, shape.keep))
    ref = {}
    for p in sorted({s % STREAM_STEPS for s in range(n)}):
        ref[p] = oracle.routing.route(xs[p].double().numpy(), wr, shape.K,
                                      oracle.routing.MODE_SOFT_PRIOR, shape.gate, prior=prior)
    near = near_order = diff_in = diff_out = 0
    c_ref = oracle.cache.SlotCache(shape.E, shape.cache_slots, "LRU")
    c_gpu = oracle.cache.SlotCache(shape.E, shape.cache_slots, "LRU")
    tot = dict(oracle_hits=0, oracle_fetches=0, replay_hits=0, replay_fetches=0)
    for s in range(n):
        p = s % STREAM_STEPS
        r, g = ref[p], idx_gpu[p]
        ho, fo, _, _ = c_ref.step(r["idx"])
        hg, fg, _, _ = c_gpu.step(g)
        if s < first:
            continue
        tot["oracle_hits"] += ho
        tot["oracle_fetches"] += fo
        tot["replay_hits"] += hg
        tot["replay_fetches"] += fg
        nk = r["gap_k"] < 1e-4
        ni = r["gap_in"] < 1e-4
        near += int(nk.sum())
        near_order += int((ni & ~nk).sum())
        differ = np.any(g != r["idx"], axis=1)
        diff_in += int((differ & (nk | ni)).sum())
        diff_out += int((differ & ~(nk | ni)).sum())
    return dict(tokens=steps * batch, near_tie_tokens=near, near_tie_rule="(s_K - s_K+1) / s_K < 1e-4",
                order_only_near_ties=near_order, ids_differ_in_band=diff_in,
                ids_differ_outside_band=diff_out, **tot)


def fetch_verdict(chk, gpu_hits, gpu_fetches):
    """fetches_exact: the GPU's counted hits and fetches over the timed steps equal the oracle's
    (routing and cache both from the oracle); cache_exact: they equal the oracle cache's on the
    GPU's own ids (the cache decision alone, independent of near ties in routing)."""
    chk = dict(chk, gpu_hits=gpu_hits, gpu_fetches=gpu_fetches)
    chk["cache_exact"] = (gpu_hits, gpu_fetches) == (chk["replay_hits"], chk["replay_fetches"])
    chk["fetches_exact"] = (gpu_hits, gpu_fetches) == (chk["oracle_hits"], chk["oracle_fetches"])
    chk["routing_exact_outside_band"] = chk["ids_differ_outside_band"] == 0
    return chk


def cpu_model():
    """The host CPU's model name (lscpu, else /proc/cpuinfo, else the platform string)."""
    import platform

    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for ln in out.splitlines():
            if ln.strip().lower().startswith("model name"):
                return ln.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        for ln in open("/proc/cpuinfo"):
            if ln.lower().startswith("model name"):
                return ln.split(":", 1)[1].strip()
    except OSError:
        pass
    return platform.processor() or platform.machine()


def oracle_timing_one_thread(shape, batch, seed, budget_s):
    """The same oracle timing in a fresh interpreter whose BLAS uses one thread. Returns
    (tokens/s, timed steps) or None if the child failed."""
    env = dict(os.environ, OPENBLAS_NUM_THREADS="1", OMP_NUM_THREADS="1", MKL_NUM_THREADS="1")
    cmd = [sys.executable, os.path.abspath(__file__), "--oracle-timing",
           json.dumps(dict(shape=shape.name, batch=batch, seed=seed, budget_s=budget_s))]
    try:
        r = subprocess.run(cmd, env=env, capture_output=True, text=True, timeout=budget_s + 300)
        d = json.loads(r.stdout.strip().splitlines()[-1])
        return d["tokens_per_s"], d["steps"]
    except (OSError, subprocess.SubprocessError, ValueError, IndexError, KeyError):
        return None


def reference_arm(args, rank, world):
    """The reference arm: there is no reference implementation to run (the paper ships no code),
    so this times the CPU oracle as it stands on the host cores, on the same workload, metric and
    unit: args.warmup untimed decode steps, then up to args.steps timed ones (each one decode step
    of 16 rows), stopping after two minutes. Under torchrun only rank 0 runs it."""
    if rank != 0:
        return 0
    shape, batch = I.MIXTRAL, 16
    seed = replica_seed(0, 0)
    lw = I.layer_weights(seed, shape)
    tps, n = oracle_decode_tokens_per_s(shape, batch, seed, budget_s=120.0, lw=lw,
                                        warmup=args.warmup, max_steps=args.steps)
    line = dict(impl="reference", metric=METRIC, value=tps, unit="tokens/s", n_gpus=args.gpus,
                steps=n, warmup=args.warmup, ms_per_step=1e3 * batch / tps, higher_is_better=True,
                scaling="weak", vs_baseline=None, dtype="f64", data="synthetic",
                config=_config(batch),
                cpu_baseline=dict(value=tps, unit="tokens/s", cores=_CORES, kind="oracle",
                                  cpu_model=cpu_model(),
                                  sample=f"{n} decode steps x batch {batch} of the same stream "
                                         f"after {args.warmup} untimed (fp64 numpy)"),
                e2e=dict(value=tps, unit="tokens/s", h2d_bytes_per_step=0, d2h_bytes_per_step=0))
    print(json.dumps(line), flush=True)
    return 0


def _config(batch):
    return {"workload": f"mixtral-8x7b-shaped MoE layer decode, batch {batch}, 512-step AR(1) "
                        "stream, soft prior keep-4-of-8, 4-slot LRU cache, host fetch",
            "d": 4096, "E": 8, "K": 2, "w": 14336, "batch": batch, "cache_slots": 4,
            "l2": "inputs larger than L2 (each step streams >= 0.7 GB of expert weights)",
            "parallelism": "replicas"}


def profile_case(case: str, dev) -> int:
    """A few forwards: the small launch sequences that ncu captures. decode16 / decode1:
    Mixtral-shaped decode at batch 16 / 1 with every expert resident (decode FFN); ds_decode1 /
    ds_decode64: the same for the DeepSeek-V2-Lite shape at batch 1 / 64; prefill / ds_prefill:
    T = 4096 tokens, hard mask keeping 4 of 8 / 48 of 64 (tcgen05 GEMMs; prefill_pair: the Mixtral
    case on CTA-pair tiles); fetch16 / ds_fetch64:
    three decode steps (Mixtral-shaped batch 16 / DeepSeek-shaped batch 64) through the cache with
    the device-driven fetch (the FFN launch that fetches its own misses / the fetch kernel)."""
    from paper_2609_34077_gb300 import mcft as M

    sh = I.DSV2_LITE if case.startswith("ds_") else I.MIXTRAL
    desc = M.desc_of(sh)
    if case in ("fetch16", "ds_fetch64"):  # decode steps with the cache, device-driven fetch
        L = DecodeLayer(sh, 16 if case == "fetch16" else 64, 7, dev)
        per_step, experts = [], []
        for s in range(3):
            before = M.mcft_cache_stats(L.cache, 0)[1]
            L.step(s, path="device")
            torch.cuda.synchronize()
            per_step.append(M.mcft_cache_stats(L.cache, 0)[1] - before)
            experts.append(len(torch.unique(L.idx[s])))
        M.mcft_device_error()
        print(json.dumps({"case": case, "fetches_per_step": per_step, "experts_per_step": experts,
                          "fetch_bytes_per_step": [n * sh.expert_bytes for n in per_step]}))
        return 0
    if case == "prefill_pair":  # the prefill case on CTA-pair tiles
        M.mcft_set_tc_tiles(M.MCFT_TC_TILES_CTA_PAIR)
        case = "prefill"
    if case in ("prefill", "ds_prefill"):  # Mixtral keeps 4 of 8, DeepSeek 48 of 64
        T, mode = 4096, M.MCFT_ROUTE_HARD_MASK
        kw = dict(mask=I.keep_mask(7, sh.E, 4 if sh is I.MIXTRAL else sh.E * 3 // 4))
        keep = [int(e) for e in np.nonzero(kw["mask"])[0]]
        x = I.hidden_iid(7, sh, T).to(dev)
    else:
        T = {"decode16": 16, "decode1": 1, "ds_decode1": 1, "ds_decode64": 64}[case]
        mode = M.MCFT_ROUTE_SOFT_PRIOR
        kw = dict(prior=I.prior_from_mask(I.keep_mask(7, sh.E, sh.keep)))
        keep = list(range(sh.E))
        x = I.ar1_streams(7, sh, 1, T)[0].to(dev)
    lw = I.layer_weights(7, sh, experts=keep)
    experts = [None if b is None else b.to(dev) for b in lw.experts]
    shared = [b.to(dev) for b in lw.shared]
    wr = lw.router.to(dev)
    ws = torch.empty(M.mcft_moe_workspace_size(desc, T), dtype=torch.uint8, device=dev)
    for _ in range(3):
        idx, gate = M.mcft_route(desc, x, wr, mode, **kw)
        y = M.mcft_moe_forward(desc, x, idx, gate, experts, shared, workspace=ws)
    M.mcft_device_error()
    torch.cuda.synchronize()
    print(json.dumps({"case": case, "T": T, "y_abs_mean": float(y.float().abs().mean())}))
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=256)
    ap.add_argument("--warmup", type=int, default=8)
    ap.add_argument("--impl", default="mcft", choices=["mcft", "reference"])
    ap.add_argument("--batch", type=int, default=16)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-extra", action="store_true", help="skip the batch-1 and prefill extras")
    ap.add_argument("--case", choices=["decode16", "decode1", "ds_decode1", "ds_decode64", "prefill",
                                       "prefill_pair", "ds_prefill", "fetch16", "ds_fetch64", "lora",
                                       "mask"],
                    help="run only a few resident-expert forwards (for profiler captures)")
    ap.add_argument("--workload", default="layer",
                    choices=["layer", "stack-mixtral", "stack-dsv2", "chain-mixtral", "chain-dsv2",
                             "lora", "mask"],
                    help="layer: the single-layer decode line; stack-*: the full decode stack "
                         "(layers on independent streams); chain-*: the chained stack; lora: the "
                         "Stage-2 LoRA forward against the plain forward (T = 4096); mask: the "
                         "Stage-1 mask sampling and gradient kernels (T = 4096)")
    ap.add_argument("--prefetch", type=int, default=0,
                    help="chain workloads: experts prefetched per layer (0 = off)")
    ap.add_argument("--policy", default="LRU", choices=["LRU", "LFU", "FIFO"])
    ap.add_argument("--graph", action="store_true", help="stack workloads: replay a captured step")
    ap.add_argument("--oracle-timing", help=argparse.SUPPRESS)  # child of oracle_timing_one_thread
    args = ap.parse_args()
    if args.oracle_timing:
        o = json.loads(args.oracle_timing)
        sh = {s_.name: s_ for s_ in (I.MIXTRAL, I.DSV2_LITE)}[o["shape"]]
        tps, n = oracle_decode_tokens_per_s(sh, o["batch"], o["seed"], budget_s=o["budget_s"])
        print(json.dumps(dict(tokens_per_s=tps, steps=n)), flush=True)
        return 0
    if args.workload in ("lora", "mask") or args.case in ("lora", "mask"):
        import __graft_entry__

        __graft_entry__.build()
        dev = torch.device("cuda", 0)
        torch.cuda.set_device(dev)
        peaks = load_peaks()
        if args.case == "lora":  # a few Mixtral-shaped Stage-2 forwards (profiler captures)
            res = run_lora(1, 1, 61, dev, peaks, shapes=(I.MIXTRAL,))
        elif args.case == "mask":
            res = run_mask(2, 1, 62, dev, peaks)
        elif args.workload == "lora":
            res = run_lora(args.steps, args.warmup, 61, dev, peaks)
        else:
            res = run_mask(args.steps, args.warmup, 62, dev, peaks)
        print(json.dumps(res), flush=True)
        return 0
    if args.workload != "layer":
        import __graft_entry__

        __graft_entry__.build()
        torch.cuda.set_device(0)
        shape, L = (I.MIXTRAL, 32) if args.workload.endswith("mixtral") else (I.DSV2_LITE, 26)
        if args.workload.startswith("chain"):
            res = run_chain(shape, L, args.steps, args.warmup, 60, torch.device("cuda", 0),
                            args.policy, args.prefetch, graph=args.graph)
        else:
            res = run_stack(shape, L, args.steps, args.warmup, 60, torch.device("cuda", 0),
                            args.policy, graph=args.graph)
        res.update(metric="masked MoE decode stack tokens/s", value=res["tokens_per_s"],
                   unit="tokens/s", higher_is_better=True, dtype="bf16", data="synthetic")
        print(json.dumps(res), flush=True)
        return 0
    if args.case:
        import __graft_entry__

        __graft_entry__.build()
        torch.cuda.set_device(0)
        return profile_case(args.case, torch.device("cuda", 0))
    rank, world, local = dist_env()
    if args.impl == "reference":
        return reference_arm(args, rank, world)
    if args.warmup < 3:
        raise SystemExit("--warmup must be >= 3")

    import __graft_entry__

    if world > 1:
        import torch.distributed as dist

        dist.init_process_group("nccl")
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    if rank == 0 or not os.path.exists(os.path.join(ROOT, "paper_2609_34077_gb300", "libmcft.so")):
        __graft_entry__.build()
    if world > 1:
        dist.barrier()
    from paper_2609_34077_gb300 import mcft as M

    M.lib()
    peaks = load_peaks()
    seed = replica_seed(0, rank)
    shape, batch = I.MIXTRAL, args.batch

    clk = ClockSampler(local)
    d, idx_main, elapsed = run_decode(shape, batch, args.steps, args.warmup, seed, dev, peaks,
                                      clocks=clk, world=world, e2e=True)
    max_el, tokens = aggregate(elapsed, batch * args.steps, world)
    link = host_link_probe(dev, shape.expert_bytes)
    ms = max_el * 1e3 / args.steps
    # the dominant kernel of the device-driven step is the one that fetches: bound by the host link
    fk = fetching_kernel(d["kernels"]) or "fetch"
    nf, msf = d["kernels"].get(fk, {}).get("launches", 0), d["kernels"].get(fk, {}).get("ms", 0.0)
    fetched = d["fetch_bytes_per_step"] * args.steps
    fetch_roof = dict(bound="host-link", kernel=fk, unit="GB/s",
                      achieved=fetched / (msf / 1e3) / 1e9 if msf else None, peak=link["best_gbs"],
                      peak_source="best pinned host-to-device rate of the link probes in this run "
                                  "(352 MB: copy engines with 1, 2, 4 concurrent copies; SM loads "
                                  "on 38, 76, 152 CTAs)",
                      traffic=None, traffic_vs=None,
                      alg_bytes_per_launch=fetched / max(1, nf), launches=nf,
                      timed_in="the profiled pass over the same steps (kernel CUDA events)")
    fetch_roof["frac"] = fetch_roof["achieved"] / link["best_gbs"] if msf else None
    if traffic_ratio(fk):  # DRAM bytes per launch, from the ncu capture's ratio
        dram_alg = fetched / max(1, nf)
        if fk == "ffn_decode_fetch":  # it also reads the step's expert weights
            dram_alg += d["ffn_dram_bytes_per_step"] * args.steps / max(1, nf)
        fetch_roof.update(traffic=traffic_ratio(fk) * dram_alg, traffic_vs=dram_alg)
    e2e = dict(d["e2e"])
    el_e2e, tok_e2e = aggregate(e2e.pop("elapsed_s"), batch * args.steps, world)
    e2e["value"] = tok_e2e / el_e2e
    line = dict(
        metric=METRIC, value=tokens / max_el, unit="tokens/s", n_gpus=world, steps=args.steps,
        warmup=args.warmup, ms_per_step=ms, higher_is_better=True,
        scaling="weak", vs_baseline=None, dtype="bf16", data="synthetic", config=_config(batch),
        roofline=fetch_roof,
        roofline_ffn=(dict(d["roofline"], note="decode FFN inside the device-driven step, sharing SMs "
                                               "and HBM with the concurrent fetch kernel")
                      if d["roofline"] else
                      dict(note="the step's FFN runs in the launch that fetches its misses, which "
                                "the host link bounds: see roofline and roofline_ffn_alone")),
        roofline_ffn_alone=d["roofline_alone"],
        kernel_gbs=d["kernel_gbs"],
        e2e=e2e, gpu_launches=d["gpu_launches"],
        gpu_launches_note="kernels launched by the same steps in the profiled pass",
        clocks=clk.summary(), kernels=d["kernels"],
        timing=dict(value="CUDA events around the timed steps, no per-kernel instrumentation",
                    profiled_ms_per_step=d["profiled_ms_per_step"],
                    passes_same_decisions=d["passes_same_decisions"]),
        cache=dict(policy="LRU", hits=d["hits"], fetches=d["fetches"], bypass=d["bypass"],
                   fetches_per_step=d["fetches_per_step"], fetches_per_token=d["fetches_per_token"],
                   hit_rate=d["hit_rate"], mean_experts_per_step=d["mean_experts_per_step"]),
        fetch=dict(path="device-driven: batches of up to 16 tokens fetch in the FFN's own launch "
                        "(its first 38 CTAs copy the misses piece by piece while the others compute "
                        "the hits, and each missed expert's items start as their pieces land); "
                        "larger batches run a fetch kernel on a copy stream beside the hits' FFN",
                   bytes_per_step=d["fetch_bytes_per_step"], host_link_probe=link,
                   link_roofline_ms_per_step=d["fetch_bytes_per_step"] / (link["best_gbs"] * 1e9) * 1e3,
                   link_frac=(d["fetch_bytes_per_step"] / (ms / 1e3)) / (link["best_gbs"] * 1e9),
                   kernel_ms_per_step=d["kernel_ms_per_step"],
                   fetch_launch_ms_per_step=d["fetch_launch_ms_per_step"],
                   step_floor=step_floor(d, link["best_gbs"], peaks["hbm"])),
        host_fetch_path=d["host_fetch_path"],
    )
    runs = {"mixtral_b%d" % batch: (shape, batch, seed, idx_main, args.steps, d)}
    if not args.no_extra:
        nb1 = min(args.steps, 256)
        b1, idx_b1, _ = run_decode(shape, 1, nb1, args.warmup, seed + 1, dev, peaks)
        b1.pop("kernels", None)
        b1["step_floor"] = step_floor(b1, link["best_gbs"], peaks["hbm"])
        b1.pop("per_step", None)
        line["batch1"] = b1
        runs["mixtral_b1"] = (shape, 1, seed + 1, idx_b1, nb1, b1)
        for bsz in (1, 8, 64):
            nds = min(args.steps, 128)
            ds, idx_ds, _ = run_decode(I.DSV2_LITE, bsz, nds, args.warmup, seed + 3, dev, peaks)
            ds.pop("kernels", None)
            ds["step_floor"] = step_floor(ds, link["best_gbs"], peaks["hbm"])
            ds.pop("per_step", None)
            line[f"dsv2_b{bsz}"] = ds
            runs[f"dsv2_b{bsz}"] = (I.DSV2_LITE, bsz, seed + 3, idx_ds, nds, ds)
        line["prefill"] = run_prefill(max(5, min(20, args.steps // 10)), 3, seed + 2, dev, peaks)
        line["stage2_lora"] = run_lora(8, 3, seed + 4, dev, peaks)
        line["stage1_mask"] = run_mask(20, 3, seed + 4, dev, peaks)
        line["read_probe"] = run_read_probe(dev, peaks)
        _BATCHES.clear()
        torch.cuda.empty_cache()
    if rank == 0 and not args.no_cpu_baseline:
        # the oracle as a checker of the timed steps: routing (near ties counted) and fetch counts
        checks = {}
        for name, (sh, bsz, sd, idx_h, n, res) in runs.items():
            chk = fetch_verdict(oracle_fetch_check(sh, bsz, sd, idx_h, args.warmup, n),
                                res["hits"], res["fetches"])
            checks[name] = chk
            if name == "mixtral_b%d" % batch:
                line["cache"]["oracle_check"] = chk
            else:
                line["batch1" if name == "mixtral_b1" else name]["oracle_check"] = chk
        line["fetches_exact"] = all(c["fetches_exact"] for c in checks.values())
        line["cache_exact"] = all(c["cache_exact"] for c in checks.values())
        line["near_tie_tokens"] = {k: c["near_tie_tokens"] for k, c in checks.items()}
        # the oracle as the timed baseline: all cores, then one thread in a fresh interpreter
        tps, n = oracle_decode_tokens_per_s(shape, batch, seed, budget_s=12.0)
        one = oracle_timing_one_thread(shape, batch, seed, 12.0)
        line["cpu_baseline"] = dict(value=tps, unit="tokens/s", cores=_CORES, kind="oracle",
                                    cpu_model=cpu_model(),
                                    sample=f"{n} decode steps x batch {batch} of the same stream "
                                           "(fp64 numpy, BLAS threads = cores)",
                                    one_thread=(dict(value=one[0], unit="tokens/s", cores=1,
                                                     sample=f"{one[1]} decode steps x batch {batch}")
                                                if one else None))
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
