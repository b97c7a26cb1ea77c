"""Benchmark of the paged tensor store on GB300.

Workload (default): the T2I intermediate handoff -- 8 GiB pool of 2 MiB pages,
64 requests in flight, each handing on bf16 text embeddings [B,512,4096],
bf16 pooled embeddings [B,768], fp32 latents [B,16,128,128] (got with the
fused fp32 -> bf16 RNE cast) and fp16 decoded images [B,3,1024,1024]; B = 8.
One step = put all 64 requests from producer buffers, get all 64 into consumer
buffers, free everything: 128 batched calls, each one kernel launch. Request
r is issued on stream r % 4 (--streams): independent requests overlap on the
GPU, the store ordering each get after its own put and each reused page after
its last reader.

Metric: algorithmic read + write bytes / time (put and get: 2 x payload,
cast get: 1.5 x the fp32 payload), GB/s, and its fraction of the measured
HBM copy rate. The inputs of one step (5.5 GiB read, 5.5 GiB written) are
far larger than L2, so no L2 flush is needed between steps.

  python bench.py [--gpus N --steps K --warmup W] [--impl reference]

Under torchrun each rank runs an independent store on its own GPU (the store
has no cross-GPU step); rank 0 prints one JSON line with the whole-job value.
"""
from __future__ import annotations

import argparse
import ctypes as C
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import workloads as W  # noqa: E402

METRIC = "batched get/put/compact GB/s (read+write bytes) and % of GB300 HBM peak"
FALLBACK_HBM_GBS = 6800.0


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=50)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", default="native", choices=["native", "reference"])
    p.add_argument("--batch", type=int, default=8, help="B of the handoff workload")
    p.add_argument("--requests", type=int, default=64)
    p.add_argument("--streams", type=int, default=4, help="streams the requests of a step are spread over")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-cpu", action="store_true")
    p.add_argument("--no-extras", action="store_true", help="skip the one-call and reclaim variants")
    p.add_argument("--no-sweep", action="store_true", help="skip timing B = 1 and B = 4")
    p.add_argument("--pool-gib", type=float, default=None, help="smaller pool (profiling small cases)")
    p.add_argument("--cpu-seconds", type=float, default=10.0, help="minimum CPU-baseline sample time")
    p.add_argument("--rows", default="tiny,unaligned,cdriver,weights,adapters,compaction,prefix,views,pull,host",
                   help="other hot-path rows timed in the same run (comma list, or 'none')")
    p.add_argument("--adapter-calls", type=int, default=10_000)
    p.add_argument("--adapter-sets", type=int, default=None, help="fewer LoRA sets (profiling small cases)")
    p.add_argument("--adapter-pool-gib", type=float, default=None, help="smaller adapter pool (profiling small cases)")
    p.add_argument("--rows-only", action="store_true", help="skip the handoff headline (profiling a row)")
    p.add_argument("--weight-blocks", type=int, default=None,
                   help="restore only the first N blocks into a pool sized for them (profiling small cases)")
    p.add_argument("--lib", default=None,
                   help="time this build of libt2istore.so instead of the package's (tuning sweeps)")
    p.add_argument("--compaction-gib", type=int, default=None,
                   help="smaller compaction pool (GiB; the limit is 3/4 of it): profiling small cases")
    return p.parse_args()


# ----------------------------------------------------------------------------- helpers
def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return FALLBACK_HBM_GBS, "fallback"


def ncu_traffic(kernel: str, launch: str):
    """dram read+write bytes of one ``kernel`` launch of shape ``launch`` from
    the committed ncu summary, if it was taken on the current kernel source
    (else None)."""
    from paper_2607_26566_gb300 import build as b

    path = os.path.join(ROOT, "profiles", "traffic.txt")
    if not os.path.exists(path):
        return None
    src_hash = b.kernel_source_hash()
    for line in open(path):
        f = dict(kv.split("=", 1) for kv in line.split() if "=" in kv)
        if f.get("kernel") == kernel and f.get("launch") == launch and f.get("source") == src_hash:
            return float(f["dram_bytes_per_launch"])
    return None


class Clocks:
    """nvidia-smi sampling of SM clocks and throttle reasons during a region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.FIELDS,
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except OSError:
            self.proc = None
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
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.lines:
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ----------------------------------------------------------------------------- handoff
class Handoff:
    """The handoff workload bound to one store. Descriptor arrays are built
    once; a step issues raw C-ABI calls only."""

    def __init__(self, B: int, requests: int, device, host_buffers: bool = False, seed: int = 0,
                 pool_bytes: int | None = None, consumers: int = 0, h2d_mode: int = 0, page_bytes: int | None = None,
                 alloc_policy: int = 0, d2h_mode: int = 0):
        import torch

        from paper_2607_26566_gb300 import Store, get_descs, put_descs

        C_ = W.HANDOFF
        self.torch = torch
        self.device = device
        self.specs = W.handoff_specs(B)
        self.n_obj = len(self.specs)
        self.requests = requests
        self.ci = W.handoff_cast_index()
        self.pool = torch.empty(pool_bytes or C_["pool_bytes"], dtype=torch.uint8, device=device)
        self.page_bytes = page_bytes or C_["page_bytes"]
        self.alloc_policy = alloc_policy
        self.store = Store(self.pool, self.page_bytes, h2d_mode=h2d_mode, alloc_policy=alloc_policy,
                           d2h_mode=d2h_mode)
        self.lib = self.store._lib
        self.h = self.store._h
        self.inputs, self.outputs = [], []
        for r in range(requests):
            ts = W.handoff_request_torch(seed, r, self.specs, device)
            outs = [torch.empty(sp.nbytes // (2 if j == self.ci else 1), dtype=torch.uint8, device=device)
                    for j, sp in enumerate(self.specs)]
            if host_buffers:
                ts = [t.cpu().pin_memory() for t in ts]
                outs = [torch.empty(o.numel(), dtype=torch.uint8).pin_memory() for o in outs]
            self.inputs.append(ts)
            self.outputs.append(outs)
        torch.cuda.synchronize(device)
        self.ids = np.zeros(requests * self.n_obj, np.uint64)
        # consumers = 1: every intermediate is reclaimed by the store after its
        # one get (§5.3) and the step issues no free
        self.consumers = consumers
        self.pd = [put_descs(ts, nbytes=[sp.nbytes for sp in self.specs], src_is_host=int(host_buffers),
                             dtype_tag=[sp.dtype_tag for sp in self.specs], consumers=consumers)
                   for ts in self.inputs]
        casts = [1 if j == self.ci else 0 for j in range(self.n_obj)]
        self.gd = [get_descs(np.zeros(self.n_obj, np.uint64), outs, cast=casts) for outs in self.outputs]
        from paper_2607_26566_gb300 import _lib as L

        # typed pointers built once: a step makes raw C-ABI calls only
        self.pd_p = [d.ctypes.data_as(C.POINTER(L.PutDesc)) for d in self.pd]
        self.gd_p = [d.ctypes.data_as(C.POINTER(L.GetDesc)) for d in self.gd]
        self.ids_p = [C.cast(C.c_void_p(self.ids.ctypes.data + 8 * self.n_obj * r), C.POINTER(C.c_uint64))
                      for r in range(requests)]
        self.all_ids_p = self.ids.ctypes.data_as(C.POINTER(C.c_uint64))
        # the CPython entry points (csrc/pycall.c) take plain integers: the
        # same calls without ctypes' per-call conversion (None: ctypes only)
        self.fast = L.pycall()
        self.pd_a = [int(d.ctypes.data) for d in self.pd]
        self.gd_a = [int(d.ctypes.data) for d in self.gd]
        self.ids_a = [int(self.ids.ctypes.data) + 8 * self.n_obj * r for r in range(requests)]
        self.hi = self.store._hi
        payload = sum(sp.nbytes for sp in self.specs)
        lat = self.specs[self.ci].nbytes
        self.put_bytes = 2 * payload * requests
        self.get_bytes = (2 * (payload - lat) + 1.5 * lat) * requests
        self.h2d_bytes = payload * requests
        self.d2h_bytes = (payload - lat // 2) * requests
        self.step_bytes = self.put_bytes + self.get_bytes

    def step(self, stream, ev=None):
        """One step. ``ev`` = three events recorded before the puts, between
        the puts and the gets, and after the gets: each phase is a run of
        back-to-back launches of one kernel."""
        if ev is not None:
            ev[0].record()
        self._puts([stream])
        if ev is not None:
            ev[1].record()
        self._gets([stream])
        if ev is not None:
            ev[2].record()
        self._free()

    def _puts(self, streams):
        """The put of every request, request r on ``streams[r % len]``
        (cudaStream_t integers)."""
        n, k, R = self.n_obj, len(streams), self.requests
        if self.fast is not None:
            put, hi, pd, ids = self.fast.put_batch, self.hi, self.pd_a, self.ids_a
            for r in range(R):
                if put(hi, pd[r], n, ids[r], streams[r % k]):
                    raise RuntimeError("put_batch: " + self.store.last_error())
            return
        lib, h = self.lib, self.h
        ss = [C.c_void_p(x) for x in streams]
        for r in range(R):
            if lib.t2i_put_batch(h, self.pd_p[r], n, self.ids_p[r], ss[r % k]):
                raise RuntimeError("put_batch: " + self.store.last_error())

    def _gets(self, streams):
        """The get of every request (with the ids of its put), request r on
        ``streams[r % len]``."""
        n, k, R = self.n_obj, len(streams), self.requests
        if self.fast is not None:
            get, hi, gd, ids = self.fast.get_batch_ids, self.hi, self.gd_a, self.ids_a
            for r in range(R):
                if get(hi, gd[r], n, ids[r], 0, streams[r % k]):
                    raise RuntimeError("get_batch: " + self.store.last_error())
            return
        lib, h = self.lib, self.h
        ss = [C.c_void_p(x) for x in streams]
        for r in range(R):
            self.gd[r]["id"] = self.ids[n * r:n * (r + 1)]
            if lib.t2i_get_batch(h, self.gd_p[r], n, None, ss[r % k]):
                raise RuntimeError("get_batch: " + self.store.last_error())

    def _free(self):
        if self.consumers:
            return
        st = (self.fast.free(self.hi, int(self.ids.ctypes.data), len(self.ids)) if self.fast is not None
              else self.lib.t2i_free(self.h, self.all_ids_p, len(self.ids)))
        if st:
            raise RuntimeError("free: " + self.store.last_error())

    def step_streams(self, streams, ev=None):
        """One step with request r on ``streams[r % k]``: independent requests
        overlap, so one launch's ramp and drain are hidden under another's
        copy. The store orders each get after its request's put (same
        stream) and each reused page after its last reader (page-level
        events), so no further synchronisation is needed; the two phases
        are still joined through ``streams[0]`` so that each phase's span is
        measurable. ``ev`` = three timing events as in :meth:`step`."""
        ss = [int(x.cuda_stream) for x in streams]
        if ev is not None:
            ev[0].record(streams[0])
        self._puts(ss)
        self._join(streams, ev[1] if ev is not None else None)
        self._gets(ss)
        self._join(streams, ev[2] if ev is not None else None)
        self._free()

    def _join(self, streams, hub_event=None):
        """Every stream waits until all of them reach this point (through
        ``streams[0]``, where ``hub_event`` is recorded)."""
        torch = self.torch
        if not hasattr(self, "_done") or len(self._done) < len(streams):
            self._done = [torch.cuda.Event() for _ in streams]
            self._hub = torch.cuda.Event()
        for x, e in zip(streams[1:], self._done):
            e.record(x)
            streams[0].wait_event(e)
        hub = hub_event if hub_event is not None else self._hub
        hub.record(streams[0])
        for x in streams[1:]:
            x.wait_event(hub)

    def step_two_streams(self, s_put, s_get):
        """The same step with puts on one stream and gets on another: the
        store orders each get after the put of its request only, so request
        r+1's put overlaps request r's get (both directions of the host link
        in the end-to-end case)."""
        n = self.n_obj
        sp, sg = int(s_put.cuda_stream), int(s_get.cuda_stream)
        if self.fast is not None:
            put, get, hi = self.fast.put_batch, self.fast.get_batch_ids, self.hi
            for r in range(self.requests):
                if put(hi, self.pd_a[r], n, self.ids_a[r], sp):
                    raise RuntimeError("put_batch: " + self.store.last_error())
                if get(hi, self.gd_a[r], n, self.ids_a[r], 0, sg):
                    raise RuntimeError("get_batch: " + self.store.last_error())
        else:
            lib, h = self.lib, self.h
            for r in range(self.requests):
                if lib.t2i_put_batch(h, self.pd_p[r], n, self.ids_p[r], C.c_void_p(sp)):
                    raise RuntimeError("put_batch: " + self.store.last_error())
                self.gd[r]["id"] = self.ids[n * r:n * (r + 1)]
                if lib.t2i_get_batch(h, self.gd_p[r], n, None, C.c_void_p(sg)):
                    raise RuntimeError("get_batch: " + self.store.last_error())
        self._free()

    def step_one_call(self):
        """The same step with one put_batch of all requests' objects and one
        get_batch of all of them (descriptors built once)."""
        if not hasattr(self, "pd_all"):
            self.pd_all = np.concatenate(self.pd)
            self.gd_all = np.concatenate(self.gd)
        st, ids = self.store.put_batch(self.pd_all)
        self.store.check(st)
        self.gd_all["id"] = ids
        st, _ = self.store.get_batch(self.gd_all, per_item=False)
        self.store.check(st)
        if not self.consumers:
            self.store.check(self.store.free(ids))

    def reopen(self, h2d_mode: int = 0, d2h_mode: int = 0, alloc_policy: int | None = None):
        """A new store over the same pool and buffers, with other host-copy
        modes or placement (after the old one's work has finished)."""
        from paper_2607_26566_gb300 import Store

        self.torch.cuda.synchronize(self.device)
        self.store.close()
        if alloc_policy is not None:
            self.alloc_policy = alloc_policy
        self.store = Store(self.pool, self.page_bytes, h2d_mode=h2d_mode, alloc_policy=self.alloc_policy,
                           d2h_mode=d2h_mode)
        self.lib = self.store._lib
        self.h = self.store._h
        self.hi = self.store._hi

    def verify(self):
        """get(put(x)) == x on every output after a step: byte equality, and
        for the cast latents equality with torch's own fp32 -> bf16 (round to
        nearest even; the N(0, 1) latents hold no NaN)."""
        torch = self.torch
        for ts, outs in zip(self.inputs, self.outputs):
            for j, (t, o) in enumerate(zip(ts, outs)):
                want = t.reshape(-1).view(torch.uint8)
                if j == self.ci:
                    want = t.reshape(-1).view(torch.float32).to(torch.bfloat16).view(torch.uint8)
                if not torch.equal(want, o.reshape(-1)):
                    raise RuntimeError("handoff output differs from its input")


def time_handoff(hw: Handoff, steps: int, warmup: int, dist_ctx, per_kernel: bool, clocks_index=None,
                 n_streams: int = 1, nvtx: str = "bench_timed"):
    """Times ``steps`` steps; with ``n_streams`` > 1 the requests of a step
    are spread over that many streams (:meth:`Handoff.step_streams`).
    ``per_kernel``: events around each phase (a run of one kernel's
    launches); returns their mean spans and the bytes they moved."""
    torch = hw.torch
    stream = torch.cuda.current_stream(hw.device)
    streams = [stream] + [torch.cuda.Stream(hw.device) for _ in range(n_streams - 1)]

    def run(ev=None):
        if n_streams == 1:
            hw.step(stream.cuda_stream, ev)
        else:
            hw.step_streams(streams, ev)

    for _ in range(warmup):
        run()
    torch.cuda.synchronize(hw.device)
    if per_kernel:
        # per step: the put phase and the get phase, each bracketed by events
        # (an event between two launches would stop the next one from starting
        # early, so single launches are not bracketed)
        evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(steps)]
    launches0 = hw.store.stats()["launches"]
    clk = Clocks(clocks_index) if clocks_index is not None else None
    if clk:
        clk.__enter__()
        time.sleep(0.3)
    dist_ctx.barrier()
    torch.cuda.synchronize(hw.device)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    torch.cuda.nvtx.range_push(nvtx)   # the headline's range is "bench_timed" (profiles filter on it)
    t0.record(stream)
    for x in streams[1:]:
        x.wait_event(t0)
    for k in range(steps):
        run(evs[k] if per_kernel else None)
    t1.record(stream)        # every stream joined stream 0 at the end of the last step
    torch.cuda.nvtx.range_pop()
    torch.cuda.synchronize(hw.device)
    dist_ctx.barrier()
    if clk:
        clk.__exit__()
    ms = t0.elapsed_time(t1)
    launches = hw.store.stats()["launches"] - launches0
    kern = None
    if per_kernel:
        # a phase holds hw.requests launches of its kernel, n_streams at a time
        put_ms = statistics.mean(e[0].elapsed_time(e[1]) for e in evs)
        get_ms = statistics.mean(e[1].elapsed_time(e[2]) for e in evs)
        steps_ms = sorted(e[0].elapsed_time(e[2]) for e in evs)
        kern = {"put_phase_ms": put_ms, "get_phase_ms": get_ms,
                "step_ms": {"median": round(statistics.median(steps_ms), 4), "best": round(steps_ms[0], 4),
                            "worst": round(steps_ms[-1], 4), "n": len(steps_ms)},
                "put_phase_bytes": hw.put_bytes, "get_phase_bytes": hw.get_bytes,
                "launches_per_phase": hw.requests, "streams": n_streams}
    return ms, launches, kern, (clk.summary() if clk else None)


def time_two_streams(hw: Handoff, steps: int, warmup: int = 2) -> float:
    """ms for ``steps`` steps with puts on one stream and gets on another
    (:meth:`Handoff.step_two_streams`), after ``warmup`` untimed steps; CUDA
    events from before the first put to after the last get."""
    torch = hw.torch
    s_put, s_get = torch.cuda.Stream(hw.device), torch.cuda.Stream(hw.device)
    for _ in range(warmup):
        hw.step_two_streams(s_put, s_get)
    torch.cuda.synchronize(hw.device)
    a, zp, zg = (torch.cuda.Event(enable_timing=True) for _ in range(3))
    a.record(s_put)
    s_get.wait_event(a)
    for _ in range(steps):
        hw.step_two_streams(s_put, s_get)
    zp.record(s_put)
    s_get.wait_event(zp)
    zg.record(s_get)
    torch.cuda.synchronize(hw.device)
    return a.elapsed_time(zg)


def time_calls(hw: Handoff, reps: int = 3) -> dict:
    """Each batched call of one step timed alone with CUDA events around it
    (one stream; an event between two launches keeps the second from
    starting early, so these are slightly slower than back to back):
    median and best over the step's 64 puts and 64 gets, ``reps`` times."""
    torch = hw.torch
    lib, h, n = hw.lib, hw.h, hw.n_obj
    stream = torch.cuda.current_stream(hw.device)
    s = C.c_void_p(stream.cuda_stream)
    hw.step(stream.cuda_stream)                                     # warm
    torch.cuda.synchronize(hw.device)
    put_ms, get_ms = [], []
    for _ in range(reps):
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(4 * hw.requests)]
        for r in range(hw.requests):
            ev[2 * r].record(stream)
            if lib.t2i_put_batch(h, hw.pd_p[r], n, hw.ids_p[r], s):
                raise RuntimeError("put_batch: " + hw.store.last_error())
            ev[2 * r + 1].record(stream)
        for r in range(hw.requests):
            hw.gd[r]["id"] = hw.ids[n * r:n * (r + 1)]
            k = 2 * hw.requests + 2 * r
            ev[k].record(stream)
            if lib.t2i_get_batch(h, hw.gd_p[r], n, None, s):
                raise RuntimeError("get_batch: " + hw.store.last_error())
            ev[k + 1].record(stream)
        torch.cuda.synchronize(hw.device)
        if lib.t2i_free(h, hw.all_ids_p, len(hw.ids)):
            raise RuntimeError("free: " + hw.store.last_error())
        put_ms += [ev[2 * r].elapsed_time(ev[2 * r + 1]) for r in range(hw.requests)]
        get_ms += [ev[2 * hw.requests + 2 * r].elapsed_time(ev[2 * hw.requests + 2 * r + 1])
                   for r in range(hw.requests)]
    pb, gb = hw.put_bytes / hw.requests, hw.get_bytes / hw.requests
    return {"calls": len(put_ms) + len(get_ms),
            "put_ms": {"median": round(statistics.median(put_ms), 5), "best": round(min(put_ms), 5)},
            "get_ms": {"median": round(statistics.median(get_ms), 5), "best": round(min(get_ms), 5)},
            "put_gbs_median": round(pb / (statistics.median(put_ms) * 1e-3) / 1e9, 1),
            "get_gbs_median": round(gb / (statistics.median(get_ms) * 1e-3) / 1e9, 1)}


class Dist:
    """Rank bookkeeping for N independent replicas (one store per GPU; the
    store has no cross-GPU step, so the only collectives are the timing
    barrier and the max / sum of the ranks' numbers)."""

    def __init__(self, backend: str | None = None, init: bool = True):
        self.world = int(os.environ.get("WORLD_SIZE", "1"))
        self.rank = int(os.environ.get("RANK", "0"))
        self.local = int(os.environ.get("LOCAL_RANK", "0"))
        self.on = self.world > 1 and init
        self.backend = None
        if self.on:
            import torch
            import torch.distributed as dist
            self.dist = dist
            self.backend = backend or ("nccl" if torch.cuda.is_available() else "gloo")
            if self.backend == "nccl":
                torch.cuda.set_device(self.local)   # each rank's collectives on its own GPU
            dist.init_process_group(self.backend)

    def barrier(self):
        if self.on:
            if self.backend == "nccl":
                self.dist.barrier(device_ids=[self.local])
            else:
                self.dist.barrier()

    def _reduce(self, x: float, op) -> float:
        if not self.on:
            return x
        import torch
        dev = f"cuda:{self.local}" if self.backend == "nccl" else "cpu"
        t = torch.tensor([x], dtype=torch.float64, device=dev)
        self.dist.all_reduce(t, op=op)
        return float(t.item())

    def max(self, x: float) -> float:
        return self._reduce(x, self.dist.ReduceOp.MAX if self.on else None)

    def sum(self, x: float) -> float:
        return self._reduce(x, self.dist.ReduceOp.SUM if self.on else None)

    def close(self):
        if self.on:
            self.dist.destroy_process_group()


def job_gbs(bytes_per_rank: float, ms_max: float, dist_ctx: "Dist") -> float:
    """Whole-job GB/s: the bytes every rank moved over the slowest rank's time."""
    return dist_ctx.sum(bytes_per_rank) / (ms_max * 1e-3) / 1e9


# ----------------------------------------------------------------------------- tiny
def time_tiny(device, reps: int = 20):
    """The tiny store: 64 MiB pool, 64 KiB pages; put 32 objects (1 KiB - 2 MiB),
    get all, free every third, put 8 more, get all 30 -- one step per rep."""
    import torch

    from paper_2607_26566_gb300 import Store, get_descs, put_descs

    C_ = W.TINY
    first, more = W.tiny_objects(0)
    src1 = [torch.from_numpy(x).to(device) for x in first]
    src2 = [torch.from_numpy(x).to(device) for x in more]
    out1 = [torch.empty_like(x) for x in src1]
    pool = torch.empty(C_["pool_bytes"], dtype=torch.uint8, device=device)
    st = Store(pool, C_["page_bytes"])
    gone_idx = W.tiny_freed_indices()
    p1, p2 = put_descs(src1), put_descs(src2)
    live_out = [o for k, o in enumerate(out1) if k not in gone_idx] + [torch.empty_like(x) for x in src2]
    # put 32 + get 32 + put 8 + get 30: read + write bytes of each
    payload = (2 * sum(x.numel() for x in src1) + 2 * sum(x.numel() for x in src2)
               + 2 * sum(x.numel() for x in src1) + 2 * sum(o.numel() for o in live_out))

    def step():
        s, ids = st.put_batch(p1)
        st.check(s)
        st.check(st.get_batch(get_descs(ids, out1), per_item=False)[0])
        st.check(st.free([int(ids[k]) for k in gone_idx]))
        s, ids2 = st.put_batch(p2)
        st.check(s)
        keep = [int(ids[k]) for k in range(len(ids)) if k not in gone_idx] + [int(i) for i in ids2]
        st.check(st.get_batch(get_descs(keep, live_out), per_item=False)[0])
        st.check(st.free(keep))

    stream = torch.cuda.current_stream(device)
    for _ in range(3):
        step()
    torch.cuda.synchronize(device)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(reps):
        step()
    e1.record(stream)
    torch.cuda.synchronize(device)
    ms = e0.elapsed_time(e1) / reps
    ok = all(torch.equal(a, b) for a, b in zip(out1, src1))
    st.close()
    return {"workload": "tiny: 64 MiB pool, 64 KiB pages, 32 + 8 uint8 objects (1 KiB - 2 MiB)",
            "ms_per_step": round(ms, 4), "gbs": round(payload / (ms * 1e-3) / 1e9, 1), "bit_exact": bool(ok),
            "launches_per_step": 4}


def time_unaligned(device, reps: int = 10, nbytes: int = 1 << 30):
    """The any-alignment kernels on one 1 GiB object (2 MiB pages, a 2 GiB
    pool): puts from sources 1, 4 and 8 bytes past a 16-byte boundary, gets
    into destinations 1 and 3 bytes past one, fp32 -> bf16 casts into
    destinations 2 and 6 bytes past one, each beside its aligned form. Every
    call is timed alone with CUDA events (median of ``reps``); the outputs of
    the last calls are compared with the input (the casts with torch's own
    round-to-nearest-even conversion)."""
    import torch

    from paper_2607_26566_gb300 import Store, get_descs, put_descs

    stream = torch.cuda.current_stream(device)
    src = torch.randn(nbytes // 4 + 16, dtype=torch.float32, device=device).view(torch.uint8)
    dst = torch.empty(nbytes + 64, dtype=torch.uint8, device=device)
    pool = torch.empty(2 << 30, dtype=torch.uint8, device=device)
    st = Store(pool, 2 << 20)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]

    def timed(fn):
        ms = []
        for _ in range(reps + 2):
            ev[0].record(stream)
            fn()
            ev[1].record(stream)
            torch.cuda.synchronize(device)
            ms.append(ev[0].elapsed_time(ev[1]))
        return statistics.median(ms[2:])

    out = {"workload": "one 1 GiB object, 2 MiB pages, user addresses at byte offsets from a 16-byte boundary",
           "reps": reps}
    ids = [0]

    def put(off):
        def fn():
            if ids[0]:
                st.check(st.free([ids[0]]))
            s, got = st.put_batch(put_descs([src.data_ptr() + off], nbytes=[nbytes]))
            st.check(s)
            ids[0] = int(got[0])
        return fn

    for off in (0, 1, 4, 8):
        out[f"put_src+{off}_gbs"] = round(2 * nbytes / (timed(put(off)) * 1e-3) / 1e9, 1)
    put(0)()  # the object now holds src[:nbytes], which the gets read back

    def get(off, cast):
        n_out = nbytes // 2 if cast else nbytes
        d = get_descs([ids[0]], [dst.data_ptr() + off], dst_bytes=[n_out], cast=cast)
        return lambda: st.check(st.get_batch(d, per_item=False)[0])

    for off in (0, 1, 3):
        out[f"get_dst+{off}_gbs"] = round(2 * nbytes / (timed(get(off, 0)) * 1e-3) / 1e9, 1)
    ok = torch.equal(dst[3:3 + nbytes], src[:nbytes])
    for off in (0, 2, 6):
        out[f"cast_dst+{off}_gbs"] = round(1.5 * nbytes / (timed(get(off, 1)) * 1e-3) / 1e9, 1)
    want = src[:nbytes].view(torch.float32).to(torch.bfloat16).view(torch.uint8)
    ok = ok and torch.equal(dst[6:6 + nbytes // 2], want)
    put(1)()
    get(1, 0)()
    torch.cuda.synchronize(device)
    ok = ok and torch.equal(dst[1:1 + nbytes], src[1:1 + nbytes])
    out["bit_exact"] = bool(ok)
    st.close()
    return out


def time_c_driver(device, steps: int = 50, warmup: int = 3):
    """The handoff step driven from C through the C ABI (cdriver/handoff_step.c,
    no Python between calls), 64 requests of 2 MiB pages in an 8 GiB pool:
    B = 1 and 8, on 4 streams and on one. Its host microseconds per call are
    the library's own cost (pointer checks, directory, page dependencies,
    launch); the gap to the Python rows is the binding's."""
    from paper_2607_26566_gb300 import build as b

    exe = b.build_cdriver()
    out = {"workload": "t2i handoff, 64 requests, 2 MiB pages, 8 GiB pool, driven from C", "runs": []}
    for B, S in ((1, 4), (1, 1), (8, 4), (8, 1)):
        r = subprocess.run([exe, str(B), "64", str(S), str(steps), str(warmup), str(2 << 20), "8", "1",
                            str(device.index or 0)], capture_output=True, text=True, timeout=600)
        if r.returncode:
            raise RuntimeError(f"C driver B={B} S={S} failed: {r.stderr.strip()[-400:]}")
        d = json.loads(r.stdout.strip().splitlines()[-1])
        if not d["outputs_ok"]:
            raise RuntimeError(f"C driver B={B} S={S}: an output differs from its input")
        out["runs"].append({k: d[k] for k in ("B", "streams", "gbs", "ms_per_step", "host_us_per_put",
                                              "host_us_per_get")})
    return out


# ----------------------------------------------------------------------------- weights
class WeightRestore:
    """Weight-cache restore: the bf16 weights of a 57-block DiT (1,140 tensors,
    11.84 B parameters, 22.05 GiB) put from pinned host memory, one put_batch
    per block (layer-wise loading), then got with one get_batch into
    contiguous per-block buffers (each tensor 256-byte aligned in its block)."""

    def __init__(self, device, seed: int = 0, h2d_mode: int = 0, n_blocks: int | None = None,
                 alloc_policy: int = 0, pool_bytes: int | None = None):
        import torch

        from paper_2607_26566_gb300 import Store, get_descs, put_descs

        C_ = W.WEIGHTS
        self.torch = torch
        self.device = device
        specs = W.dit_weight_specs()
        layout = W.block_layout(specs)
        if n_blocks is not None:
            layout = layout[:n_blocks]
        self.specs, self.layout = specs, layout
        if pool_bytes is None and n_blocks is not None:
            # room for the blocks' pages (each tensor rounded up to whole pages)
            P = C_["page_bytes"]
            pool_bytes = sum(-(-specs[i].nbytes // P) * P for _, members in layout for i, _ in members)
        self.pool = torch.empty(pool_bytes or C_["pool_bytes"], dtype=torch.uint8, device=device)
        self.store = Store(self.pool, C_["page_bytes"], h2d_mode=h2d_mode, alloc_policy=alloc_policy)
        self.host = []      # pinned per-block source buffers
        self.dst = []       # device per-block destination buffers
        for total, members in layout:
            d = torch.empty(total, dtype=torch.uint8, device=device)
            for i, off in members:
                v = W.weight_values_torch(seed, i, specs[i], device)
                d[off:off + specs[i].nbytes].copy_(v.view(torch.uint8))
            h = torch.empty(total, dtype=torch.uint8).pin_memory()
            h.copy_(d)
            d.fill_(0xA5)
            self.host.append(h)
            self.dst.append(d)
        torch.cuda.synchronize(device)
        self.pd = []
        all_dst, all_bytes = [], []
        for b, (total, members) in enumerate(layout):
            base = self.host[b].data_ptr()
            self.pd.append(put_descs([base + off for _, off in members], nbytes=[specs[i].nbytes for i, _ in members],
                                     src_is_host=1, dtype_tag=W.DTYPE_BF16, group=0, order=b, evictable=1))
            all_dst += [self.dst[b].data_ptr() + off for _, off in members]
            all_bytes += [specs[i].nbytes for i, _ in members]
        self.n_tensors = len(all_dst)
        self.gd = get_descs(np.zeros(self.n_tensors, np.uint64), all_dst, dst_bytes=all_bytes)
        self.payload = sum(all_bytes)
        self.ids = None

    def put_all(self):
        ids = []
        for d in self.pd:
            st, i = self.store.put_batch(d)
            self.store.check(st)
            ids.append(i)
        self.ids = np.concatenate(ids)
        self.gd["id"] = self.ids

    def get_all(self):
        st, _ = self.store.get_batch(self.gd, per_item=False)
        self.store.check(st)

    def free_all(self):
        self.store.check(self.store.free(self.ids))
        self.ids = None

    def verify(self) -> bool:
        torch = self.torch
        return all(torch.equal(h.to(self.device, non_blocking=False), d) for h, d in zip(self.host, self.dst))

    def close(self):
        self.store.close()


def time_weights(device, reps: int = 3, h2d_mode: int = 0, n_blocks: int | None = None):
    import torch

    wr = WeightRestore(device, h2d_mode=h2d_mode, n_blocks=n_blocks)
    stream = torch.cuda.current_stream(device)
    wr.put_all()
    wr.get_all()
    wr.free_all()
    torch.cuda.synchronize(device)
    e = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
    put_ms, get_ms, get_kern_ms = [], [], []
    launches0 = wr.store.stats()["launches"]
    for _ in range(reps):
        e[0].record(stream)
        wr.put_all()
        e[1].record(stream)
        wr.get_all()
        e[2].record(stream)
        torch.cuda.synchronize(device)
        put_ms.append(e[0].elapsed_time(e[1]))
        get_ms.append(e[1].elapsed_time(e[2]))
        gate(device)   # the same get behind a gate: its launches alone
        e[1].record(stream)
        wr.get_all()
        e[2].record(stream)
        torch.cuda.synchronize(device)
        get_kern_ms.append(e[1].elapsed_time(e[2]))
        wr.free_all()
    launches = (wr.store.stats()["launches"] - launches0) / reps
    ok = wr.verify()
    pm, gm, gk = statistics.median(put_ms), statistics.median(get_ms), statistics.median(get_kern_ms)
    # the host link's ceiling on this machine: a plain pinned copy (torch) of 1 GiB
    hb = torch.empty(1 << 30, dtype=torch.uint8).pin_memory()
    db = torch.empty(1 << 30, dtype=torch.uint8, device=device)
    db.copy_(hb, non_blocking=True)
    torch.cuda.synchronize(device)
    e[0].record(stream)
    for _ in range(3):
        db.copy_(hb, non_blocking=True)
    e[1].record(stream)
    torch.cuda.synchronize(device)
    link_ceiling = 3 * (1 << 30) / (e[0].elapsed_time(e[1]) * 1e-3) / 1e9
    del hb, db
    out = {"workload": ("weight restore: 57-block DiT, 1,140 bf16 tensors, 40 GiB pool, 2 MiB pages" if n_blocks is None
                        else f"weight restore (small case): the first {n_blocks} blocks, {wr.n_tensors} tensors"),
           "payload_bytes": int(wr.payload), "h2d_mode": h2d_mode,
           "h2d_put_ms": round(pm, 3), "h2d_link_gbs": round(wr.payload / (pm * 1e-3) / 1e9, 1),
           "pinned_copy_ceiling_gbs": round(link_ceiling, 1),
           "h2d_frac_of_pinned_copy": round(wr.payload / (pm * 1e-3) / 1e9 / link_ceiling, 3),
           "h2d_vs_pcie_gen5_x16_64gbs": round(wr.payload / (pm * 1e-3) / 1e9 / 64.0, 2),
           "get_call_ms": round(gm, 3), "get_call_gbs": round(2 * wr.payload / (gm * 1e-3) / 1e9, 1),
           "get_kernel_ms": round(gk, 3), "get_gbs": round(2 * wr.payload / (gk * 1e-3) / 1e9, 1),
           "launches_per_rep": launches, "bit_exact": bool(ok)}
    wr.close()
    del wr
    torch.cuda.empty_cache()
    return out


# ----------------------------------------------------------------------------- adapters
class Adapters:
    """Multi-tenant adapter cache: 512 LoRA sets (836 bf16 objects each) behind
    a 16 GiB pool of 256 KiB pages; each call gets a window of 256 objects of a
    Zipf(1.1)-popular set. Objects of a set that are not resident (never
    loaded, or evicted: the last layers of the least recently used sets go
    first, §5.3) are put again from pinned host memory before the get -- only
    the missing ones, so a set's surviving first layers are reused."""

    def __init__(self, device, seed: int = 0, n_sets: int = 512, n_calls: int = 10_000,
                 pool_bytes: int | None = None, window: int = 256, alloc_policy: int = 0):
        import torch

        from paper_2607_26566_gb300 import Store, get_descs, put_descs

        C_ = W.ADAPTERS
        self.torch = torch
        self.device = device
        self.get_descs, self.put_descs = get_descs, put_descs
        self.window = window
        self.ranks = W.lora_ranks(seed, n_sets)
        self.objs = {r: W.lora_objects(int(r)) for r in set(int(x) for x in self.ranks)}
        self.sizes = {r: np.array([n for _, n in o], np.int64) for r, o in self.objs.items()}
        self.blocks = {r: np.array([b for b, _ in o], np.int64) for r, o in self.objs.items()}
        self.rel = {r: np.concatenate([[0], np.cumsum(v)[:-1]]) for r, v in self.sizes.items()}
        set_bytes = np.array([self.sizes[int(r)].sum() for r in self.ranks], np.int64)
        self.bank_bytes = int(set_bytes.max() + (1 << 20))
        bank = W.lora_bank_torch(seed, self.bank_bytes, device)
        self.bank = torch.empty(self.bank_bytes, dtype=torch.uint8).pin_memory()
        self.bank.copy_(bank)
        self.bank_dev = bank   # kept for verification
        self.off = W.lora_bank_offsets(seed, set_bytes, self.bank_bytes)
        self.sets, self.starts = W.adapter_calls(seed, n_calls, n_sets, 836, window, C_["zipf_s"])
        self.pool = torch.empty(pool_bytes or C_["pool_bytes"], dtype=torch.uint8, device=device)
        self.store = Store(self.pool, C_["page_bytes"], alloc_policy=alloc_policy)
        max_window = max(int(np.sort(v)[::-1][:window].sum()) for v in self.sizes.values())
        self.dst = torch.empty(max_window, dtype=torch.uint8, device=device)
        self.ids = {}          # set -> ids of its objects (stale where evicted)
        self.missing = {}      # set -> object indices evicted since their put
        self.owner = {}        # live id -> (set, object index)
        self.loads = 0
        self.load_bytes = 0
        self.load_objects = 0
        self.window_misses = 0
        self.got_bytes = 0
        self.calls_done = 0
        self.victims = []      # every eviction, in order (for comparison with the oracle)
        self.load_events = None  # a list: events around every reload put (timing)

    def load(self, s: int):
        """Puts the missing objects of set s (all of them the first time)."""
        r = int(self.ranks[s])
        if s not in self.ids:
            js = np.arange(len(self.sizes[r]))
            self.ids[s] = np.zeros(len(js), np.uint64)
        else:
            js = np.array(sorted(self.missing.get(s, ())), np.int64)
            if len(js) == 0:
                return
        base = self.bank.data_ptr() + int(self.off[s])
        d = self.put_descs(base + self.rel[r][js], nbytes=self.sizes[r][js], src_is_host=1,
                           dtype_tag=W.DTYPE_BF16, group=s, order=self.blocks[r][js], evictable=1)
        if self.load_events is not None:
            ev = (self.torch.cuda.Event(enable_timing=True), self.torch.cuda.Event(enable_timing=True))
            ev[0].record()
        st, ids = self.store.put_batch(d)
        self.store.check(st)
        if self.load_events is not None:
            ev[1].record()
            self.load_events.append(ev)
        self.ids[s][js] = ids
        self.missing[s] = set()
        for j, i in zip(js, ids):
            self.owner[int(i)] = (s, int(j))
        for v in self.store.ctl.last_evictions():
            s2, j2 = self.owner.pop(v)
            self.missing.setdefault(s2, set()).add(j2)
            self.victims.append(v)
        self.loads += 1
        self.load_objects += len(js)
        self.load_bytes += int(self.sizes[r][js].sum())

    def descs(self, k: int):
        s, w = int(self.sets[k]), int(self.starts[k])
        r = int(self.ranks[s])
        sz = self.sizes[r][w:w + self.window]
        dst_rel = np.concatenate([[0], np.cumsum(sz)[:-1]])
        return s, w, self.get_descs(self.ids[s][w:w + self.window], self.dst.data_ptr() + dst_rel, dst_bytes=sz)

    def call(self, k: int, stream=None):
        s, w = int(self.sets[k]), int(self.starts[k])
        if s not in self.ids or any(w <= j < w + self.window for j in self.missing.get(s, ())):
            self.window_misses += 1
            self.load(s)
        s, w, d = self.descs(k)
        st, _ = self.store.get_batch(d, stream=stream, per_item=False)
        self.store.check(st)
        self.got_bytes += int(d["dst_bytes"].sum())
        self.calls_done += 1
        return s, w

    def expected(self, s: int, w: int):
        """The window's bytes as the oracle's get returns them: the set's
        objects are the bank window at the set's offset, in object order."""
        r = int(self.ranks[s])
        a = int(self.off[s]) + int(self.rel[r][w])
        n = int(self.sizes[r][w:w + self.window].sum())
        return self.bank_dev[a:a + n]

    def close(self):
        self.store.close()


def time_adapters(device, n_calls: int = 10_000, check_every: int = 500, n_sets: int | None = None,
                  pool_bytes: int | None = None):
    import torch

    ad = Adapters(device, n_calls=n_calls, n_sets=n_sets or W.ADAPTERS["n_sets"], pool_bytes=pool_bytes)
    ad.load_events = []
    stream = torch.cuda.current_stream(device)
    torch.cuda.synchronize(device)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s0 = ad.store.stats()
    t_wall = time.perf_counter()
    e0.record(stream)
    bad = 0
    for k in range(n_calls):
        s, w = ad.call(k)
        if check_every and k % check_every == 0:
            n = ad.expected(s, w).numel()
            bad += int(not torch.equal(ad.dst[:n], ad.expected(s, w)))
    e1.record(stream)
    torch.cuda.synchronize(device)
    wall = time.perf_counter() - t_wall
    ms = e0.elapsed_time(e1)
    s1 = ad.store.stats()
    load_ms = sum(a.elapsed_time(b) for a, b in ad.load_events)
    # the hit path alone: the same calls again with every set resident
    # (no misses are possible once a call's set has just been touched)
    hits_ms, hit_bytes, hit_calls = 0.0, 0, 0
    h0, h1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    # a set is whole while its first victim (last object: highest layer,
    # highest id) is live
    whole = {s for s, ids in ad.ids.items() if ad.store.ctl.object(int(ids[-1]))[0] == 0}
    resident = [k for k in range(n_calls) if int(ad.sets[k]) in whole][:2000]
    ok_desc = [ad.descs(k)[2] for k in resident]
    for d in ok_desc[:20]:
        ad.store.check(ad.store.get_batch(d, per_item=False)[0])
    torch.cuda.synchronize(device)
    # raw C-ABI calls with descriptor arrays built beforehand: this times the
    # library, not the Python binding's per-call conversions
    from paper_2607_26566_gb300 import _lib as L
    lib, h, s_h = ad.store._lib, ad.store._h, C.c_void_p(stream.cuda_stream)
    ptrs = [d.ctypes.data_as(C.POINTER(L.GetDesc)) for d in ok_desc]
    sizes = [int(d["dst_bytes"].sum()) for d in ok_desc]
    h0.record(stream)
    t_hit = time.perf_counter()
    for d, pt, nb in zip(ok_desc, ptrs, sizes):
        st = lib.t2i_get_batch(h, pt, len(d), None, s_h)
        if st:
            break
        hit_bytes += nb
        hit_calls += 1
    h1.record(stream)
    torch.cuda.synchronize(device)
    t_hit = time.perf_counter() - t_hit
    hits_ms = h0.elapsed_time(h1)
    # the same hit calls with call k on stream k % 4, each stream with its own
    # destination buffer (four consumers): the gets only read shared pages
    streams = [stream] + [torch.cuda.Stream(device) for _ in range(3)]
    bufs = [ad.dst] + [torch.empty_like(ad.dst) for _ in range(3)]
    desc4 = []
    for k, d in enumerate(ok_desc):
        d4 = d.copy()
        d4["dst"] += np.uint64(bufs[k % 4].data_ptr() - ad.dst.data_ptr())
        desc4.append(d4)
    ptr4 = [d.ctypes.data_as(C.POINTER(L.GetDesc)) for d in desc4]
    ss = [C.c_void_p(x.cuda_stream) for x in streams]
    h0.record(stream)
    for x in streams[1:]:
        x.wait_event(h0)
    n4 = 0
    for k, (d, pt) in enumerate(zip(desc4, ptr4)):
        if lib.t2i_get_batch(h, pt, len(d), None, ss[k % 4]):
            break
        n4 += 1
    for x in streams[1:]:
        ev = torch.cuda.Event()
        ev.record(x)
        stream.wait_event(ev)
    h1.record(stream)
    torch.cuda.synchronize(device)
    hits4_ms = h0.elapsed_time(h1)
    hit4_bytes = sum(sizes[:n4])
    small = n_sets is not None or pool_bytes is not None
    out = {"workload": ("adapters: 512 LoRA sets (ranks 8-64), 16 GiB pool, 256 KiB pages, Zipf(1.1), 256-object gets"
                        if not small else f"adapters (small case): {len(ad.ranks)} sets, "
                                          f"{ad.pool.numel() / 2**30:.1f} GiB pool"),
           "calls": n_calls, "ms": round(ms, 2), "calls_per_s": round(n_calls / (ms * 1e-3), 1),
           "wall_calls_per_s": round(n_calls / wall, 1),
           "window_misses": ad.window_misses, "reloads": ad.loads, "reloaded_objects": ad.load_objects,
           "load_gib": round(ad.load_bytes / 2**30, 2), "evictions": int(s1["evictions"] - s0["evictions"]),
           "miss_h2d_ms": round(load_ms, 2), "miss_h2d_link_gbs": round(ad.load_bytes / (load_ms * 1e-3) / 1e9, 1),
           "miss_share_of_time": round(load_ms / ms, 4),
           "all_calls_gbs": round((2 * ad.got_bytes + ad.load_bytes) / (ms * 1e-3) / 1e9, 1),
           "hit_calls": hit_calls, "hit_gbs": round(2 * hit_bytes / (hits_ms * 1e-3) / 1e9, 1),
           "hit_calls_per_s": round(hit_calls / (hits_ms * 1e-3), 1),
           "hit_host_calls_per_s": round(hit_calls / t_hit, 1),
           "hit_streams4_gbs": round(2 * hit4_bytes / (hits4_ms * 1e-3) / 1e9, 1),
           "hit_streams4_calls_per_s": round(n4 / (hits4_ms * 1e-3), 1),
           "checked_windows_bad": bad}
    ad.close()
    del ad
    torch.cuda.empty_cache()
    return out


# ----------------------------------------------------------------------------- compaction
class Compaction:
    """Compaction under reclaim: a 64 GiB pool of 2 MiB pages fragmented by
    the seeded alloc/free trace to ~50% occupancy (objects that die in the
    trace are reserve puts; survivors carry bytes from a device bank), then
    compact(48 GiB) to hand a contiguous 16 GiB tail back."""

    def __init__(self, device, seed: int = 1, pool_bytes: int | None = None, limit_bytes: int | None = None,
                 n_ops: int | None = None, hi: int | None = None):
        import torch

        from paper_2607_26566_gb300 import put_descs

        C_ = W.COMPACTION
        self.torch = torch
        self.device = device
        self.put_descs = put_descs
        self.P = C_["page_bytes"]
        self.pool_bytes = pool_bytes or C_["pool_bytes"]
        self.limit = limit_bytes or C_["limit_bytes"]
        self.trace = W.compaction_trace(seed, self.pool_bytes // self.P, self.P, n_ops or C_["n_ops"], C_["lo"],
                                        hi or C_["hi"], C_["p_free"], C_["settle_frac"])
        self.bank_bytes = (hi or C_["hi"]) + (1 << 20)
        g = torch.Generator(device=device)
        g.manual_seed(seed * 31 + 5)
        self.bank = torch.randint(0, 256, (self.bank_bytes,), dtype=torch.uint8, device=device, generator=g)
        rng = W.rng(seed, 7)
        self.off = {k: int(rng.integers(0, (self.bank_bytes - self.trace.sizes[k]) // 256 + 1)) * 256
                    for k in self.trace.survivors}
        self.pool = torch.empty(self.pool_bytes, dtype=torch.uint8, device=device)
        self.store = None

    def build(self):
        from paper_2607_26566_gb300 import Store

        if self.store is not None:
            self.store.close()
        self.store = Store(self.pool, self.P)
        surv = set(self.trace.survivors)
        ids = {}
        bank = self.bank.data_ptr()
        for op in self.trace.ops:
            if op[0] == "alloc":
                k, n = op[1], op[2]
                src = bank + self.off[k] if k in surv else 0
                st, i = self.store.put_batch(self.put_descs([src], nbytes=[n]))
                self.store.check(st)
                ids[k] = int(i[0])
            else:
                self.store.check(self.store.free([ids.pop(op[1])]))
        self.ids = ids
        self.torch.cuda.synchronize(self.device)

    def verify(self) -> bool:
        """Every survivor got back and compared with its bank window."""
        torch = self.torch
        from paper_2607_26566_gb300 import get_descs

        n_max = max(self.trace.sizes[k] for k in self.ids)
        buf = torch.empty(n_max, dtype=torch.uint8, device=self.device)
        for k, i in self.ids.items():
            n = self.trace.sizes[k]
            self.store.check(self.store.get_batch(get_descs([i], [buf.data_ptr()], dst_bytes=[n]), per_item=False)[0])
            if not torch.equal(buf[:n], self.bank[self.off[k]:self.off[k] + n]):
                return False
        return True

    def close(self):
        if self.store is not None:
            self.store.close()


def gate(device, ms: float = 20.0):
    """Occupy the stream for ``ms`` with torch's bounded sleep kernel, so that
    the host work of the next call (planning, descriptor packing) happens
    while the GPU is busy and events after the gate time the kernels alone."""
    import torch

    torch.cuda._sleep(int(ms * 1e-3 * 2.0e9))


def time_compaction(device, reps: int = 2, pool_gib: int | None = None):
    """Call-level time (events around t2i_compact with an idle GPU, so the
    host's planning is included) and kernel-level time (the same call behind a
    gate: the compaction launches alone), each the median of ``reps``."""
    import torch

    if pool_gib:
        cp = Compaction(device, pool_bytes=pool_gib << 30, limit_bytes=(pool_gib << 30) * 3 // 4,
                        n_ops=max(2000, 100_000 * pool_gib // 64), hi=min(W.COMPACTION["hi"], (pool_gib << 30) // 128))
    else:
        cp = Compaction(device)
    stream = torch.cuda.current_stream(device)
    call_ms, kern_ms, moved_b, moved_p, launches = [], [], 0, 0, 0
    for r in range(2 * reps + 1):
        cp.build()
        gated = r % 2 == 1
        s0 = cp.store.stats()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize(device)
        if gated:
            gate(device)
        e0.record(stream)
        st, moved = cp.store.compact(cp.limit)
        e1.record(stream)
        torch.cuda.synchronize(device)
        cp.store.check(st)
        s1 = cp.store.stats()
        if r:  # the first repetition warms up
            (kern_ms if gated else call_ms).append(e0.elapsed_time(e1))
        moved_b = s1["bytes_moved"] - s0["bytes_moved"]
        moved_p = moved
        launches = s1["launches"] - s0["launches"]
    ok = cp.verify()
    cm, km = statistics.median(call_ms), statistics.median(kern_ms)
    out = {"workload": ("compaction: 64 GiB pool, 2 MiB pages, 100,000-op trace, compact to 48 GiB" if not pool_gib
                        else f"compaction (small case): {pool_gib} GiB pool, compact to 3/4"),
           "pages_moved": int(moved_p), "bytes_moved": int(moved_b), "launches": int(launches),
           "kernel_ms": round(km, 3), "gbs": round(2 * moved_b / (km * 1e-3) / 1e9, 1),
           "call_ms": round(cm, 3), "call_gbs": round(2 * moved_b / (cm * 1e-3) / 1e9, 1),
           "live_objects": len(cp.ids), "bit_exact": bool(ok)}
    cp.close()
    del cp
    torch.cuda.empty_cache()
    return out


# ----------------------------------------------------------------------------- prefix caching
class PrefixPipeline:
    """First-layer prefix caching (§5.1) on the 57-block DiT: the first L_e
    blocks stay in the store; on a request the rest stream from pinned host
    memory (copy engine, one t2i_put_layers on a load stream, an event per
    block) while a compute stream takes each block out of the store
    (t2i_get_batch_after on its event) and runs a synthetic inference of
    T_comp per block (torch's bounded sleep kernel)."""

    def __init__(self, device, n_blocks: int | None = None, load_to_comp: float = 3.2, seed: int = 0):
        import torch

        from paper_2607_26566_gb300 import get_descs

        self.torch = torch
        self.device = device
        # extent placement: each tensor lands on consecutive pages, one copy-engine copy per tensor
        self.wr = WeightRestore(device, seed=seed, h2d_mode=1, n_blocks=n_blocks, alloc_policy=1)
        self.store = self.wr.store
        self.L = len(self.wr.layout)
        self.off = np.zeros(self.L + 1, np.uint32)
        for b, d in enumerate(self.wr.pd):
            self.off[b + 1] = self.off[b] + len(d)
        self.descs = np.concatenate(self.wr.pd)
        self.work = torch.empty(max(t for t, _ in self.wr.layout), dtype=torch.uint8, device=device)
        self.s_load = torch.cuda.Stream(device)
        self.s_comp = torch.cuda.Stream(device)
        self.ids = np.zeros(len(self.descs), np.uint64)
        self.get_descs = get_descs
        self.load_to_comp = load_to_comp
        self.cycles_per_ms = None

    def _layer_gd(self, b):
        lo, hi = int(self.off[b]), int(self.off[b + 1])
        rel = [0]
        for n in self.descs["nbytes"][lo:hi][:-1]:
            rel.append(rel[-1] + int((int(n) + 255) // 256 * 256))
        return self.get_descs(self.ids[lo:hi], self.work.data_ptr() + np.array(rel, np.uint64),
                              dst_bytes=self.descs["nbytes"][lo:hi])

    def free_all(self):
        live = [int(i) for i in self.ids if int(i)]
        if live:
            self.store.check(self.store.free(live))
        self.ids[:] = 0

    def calibrate(self):
        """Per-block load times (events between consecutive blocks of one
        streamed load) and per-block get times; the sleep kernel's rate."""
        torch = self.torch
        for rep in range(2):   # the first streamed load warms the host link and the pinned pages up
            self.free_all()
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(self.L + 1)]
            ev[0].record(self.s_load)
            st, ids = self.store.put_layers(self.descs, self.off, 0, stream=self.s_load, events=ev[1:])
            self.store.check(st)
            self.ids[:] = ids
            torch.cuda.synchronize(self.device)
        self.t_load = [ev[b].elapsed_time(ev[b + 1]) for b in range(self.L)]
        g = [torch.cuda.Event(enable_timing=True) for _ in range(self.L + 1)]
        g[0].record(self.s_comp)
        for b in range(self.L):
            self.store.check(self.store.get_batch(self._layer_gd(b), stream=self.s_comp, per_item=False)[0])
            g[b + 1].record(self.s_comp)
        torch.cuda.synchronize(self.device)
        self.t_get = [g[b].elapsed_time(g[b + 1]) for b in range(self.L)]
        a, z = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(self.s_comp):
            a.record()
            torch.cuda._sleep(int(20e6))
            z.record()
        torch.cuda.synchronize(self.device)
        self.cycles_per_ms = 20e6 / a.elapsed_time(z)
        mean_load = sum(self.t_load) / self.L
        self.t_sleep = mean_load / self.load_to_comp
        self.free_all()

    def request(self, L_e: int, load_times: list | None = None):
        """One request with the first L_e blocks cached; returns ms. With
        ``load_times`` (a list), the per-block load times of this request
        (between consecutive block events on the load stream) are appended."""
        torch = self.torch
        self.free_all()
        st, ids = self.store.put_layers(self.descs, self.off[:L_e + 1], 0, stream=self.s_comp)
        self.store.check(st)
        n = int(self.off[L_e])
        self.ids[:n] = ids[:n]
        torch.cuda.synchronize(self.device)
        ev = [torch.cuda.Event(enable_timing=load_times is not None) for _ in range(self.L)]
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        # the request arrives at t0: loading and inference start together (a
        # 20 ms gate on the compute stream lets the host queue everything first)
        with torch.cuda.stream(self.s_comp):
            torch.cuda._sleep(int(20 * self.cycles_per_ms))
        t0.record(self.s_comp)
        self.s_load.wait_event(t0)
        st, ids = self.store.put_layers(self.descs, self.off, L_e, stream=self.s_load, events=ev)
        self.store.check(st)
        lo = int(self.off[L_e])
        self.ids[lo:] = ids[lo:]
        cycles = int(self.t_sleep * self.cycles_per_ms)
        for b in range(self.L):
            self.store.check(self.store.get_batch(self._layer_gd(b), stream=self.s_comp, per_item=False,
                                                  wait_event=ev[b] if b >= L_e else None)[0])
            with torch.cuda.stream(self.s_comp):
                torch.cuda._sleep(cycles)
        t1.record(self.s_comp)
        torch.cuda.synchronize(self.device)
        if load_times is not None:
            prev = t0
            for b in range(L_e, self.L):
                load_times.append(prev.elapsed_time(ev[b]))
                prev = ev[b]
        return t0.elapsed_time(t1)

    def close(self):
        self.wr.close()


def time_prefix(device, n_blocks: int | None = None, reps: int = 3):
    """ppl.(0): nothing cached, every block streamed while the blocks compute;
    its per-block load times (measured inside that request) feed the
    pipeline model, which gives the prefix L_e' that hides loading; then
    requests with L_e'/2, L_e' and all blocks cached."""
    from paper_2607_26566_gb300 import e2e_latency, pipeline_latency, prefix_layers, prefix_layers_pipeline

    pp = PrefixPipeline(device, n_blocks=n_blocks)
    pp.calibrate()
    L = pp.L
    comp = [pp.t_sleep + g for g in pp.t_get]          # per block on the compute stream
    runs, loads = {}, None
    for _ in range(reps):
        lt = []
        ms = pp.request(0, load_times=lt)
        if "0" not in runs or ms < runs["0"]:
            runs["0"], loads = ms, lt
    le_star = prefix_layers_pipeline(loads, comp)
    mean_load, mean_comp = sum(loads) / L, sum(comp) / L
    le_eq2 = prefix_layers(L, mean_load, mean_comp)
    for L_e in sorted({le_star // 2, le_star, L}):
        runs[str(L_e)] = min(pp.request(L_e) for _ in range(reps))
    out = {"workload": f"prefix caching: {L}-block DiT weights from pinned host (copy engine, extent placement), "
                       f"T_comp = 1/{pp.load_to_comp} of the mean calibration load time per block",
           "blocks": L, "t_load_ms_mean": round(mean_load, 4), "t_comp_ms_mean": round(mean_comp, 4),
           "prefix_pipeline": le_star, "prefix_eq2_means": le_eq2, "compute_only_ms": round(sum(comp), 3),
           "runs": {}}
    base = runs["0"] - sum(comp)
    for k in sorted(runs, key=int):
        L_e, ms = int(k), runs[k]
        exposed = ms - sum(comp)
        out["runs"][k] = {"measured_ms": round(ms, 3),
                          "pipeline_model_ms": round(pipeline_latency(loads, comp, L_e), 3),
                          "eq1_ms": round(e2e_latency(L, L_e, mean_load, mean_comp), 3),
                          "exposed_loading_ms": round(exposed, 3),
                          "loading_reduction_vs_ppl0": round(1 - exposed / base, 3) if base > 0 else None}
    pp.close()
    return out


# ----------------------------------------------------------------------------- views
def contiguous_fraction(store, ids) -> tuple[float, int]:
    """Fraction of the live multi-page objects among ``ids`` whose pages are
    consecutive (those a view can serve), and how many were looked at."""
    n = ok = 0
    for i in ids:
        st, info, pages = store.ctl.object(int(i))
        if st != 0 or len(pages) < 2:
            continue
        n += 1
        ok += all(pages[j] == pages[0] + j for j in range(len(pages)))
    return (ok / n if n else 1.0), n


def time_views(device, adapter_calls: int = 3000):
    """Zero-copy views: the weight restore with extent placement (every tensor
    viewed in place instead of copied out), and how contiguous the adapter
    cache stays under each placement policy after eviction churn."""
    import torch

    out = {"workload": "views: weight restore (extent placement) and adapter-cache contiguity per policy"}
    wr = WeightRestore(device, alloc_policy=1)
    wr.put_all()
    torch.cuda.synchronize(device)
    t = time.perf_counter()
    ok = 0
    for i in wr.ids:
        ok += wr.store.view(int(i))[0] == 0
    dt = time.perf_counter() - t
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    wr.get_all()
    e1.record()
    torch.cuda.synchronize(device)
    out["weights_viewable"] = f"{ok}/{len(wr.ids)}"
    out["weights_view_host_us"] = round(1e6 * dt / len(wr.ids), 2)
    out["weights_all_views_ms"] = round(1e3 * dt, 3)
    out["weights_copy_get_ms"] = round(e0.elapsed_time(e1), 3)
    wr.close()
    del wr
    torch.cuda.empty_cache()
    for policy in (0, 1):
        ad = Adapters(device, n_calls=adapter_calls, alloc_policy=policy)
        for k in range(adapter_calls):
            ad.call(k)
        ids = list(ad.owner)
        frac, n = contiguous_fraction(ad.store, ids)
        out[f"adapters_policy{policy}_contiguous"] = round(frac, 4)
        out[f"adapters_policy{policy}_multipage_objects"] = n
        ad.close()
        del ad
        torch.cuda.empty_cache()
    return out


# ----------------------------------------------------------------------------- pull
def time_pull(device, B: int = 8, requests: int = 64, reps: int = 3):
    """Producer -> consumer store pulls (§5.2) of the handoff intermediates:
    one t2i_pull per request, page to page, then the consumer frees them."""
    import torch

    from paper_2607_26566_gb300 import Store

    hw = Handoff(B, requests, device)
    stream = torch.cuda.current_stream(device)
    cons_pool = torch.empty(W.HANDOFF["pool_bytes"], dtype=torch.uint8, device=device)
    cons = Store(cons_pool, W.HANDOFF["page_bytes"])
    n = hw.n_obj
    for r in range(requests):     # the producers' outputs
        st, ids = hw.store.put_batch(hw.pd[r])
        hw.store.check(st)
        hw.ids[n * r:n * (r + 1)] = ids
    payload = sum(sp.nbytes for sp in hw.specs) * requests

    # raw C-ABI calls with arrays built once (the binding's per-call array
    # allocations would make the host, not the GPU, the bottleneck)
    lib = cons._lib
    new = np.zeros(requests * n, np.uint64)
    src_p = [C.cast(C.c_void_p(hw.ids.ctypes.data + 8 * n * r), C.POINTER(C.c_uint64)) for r in range(requests)]
    dst_p = [C.cast(C.c_void_p(new.ctypes.data + 8 * n * r), C.POINTER(C.c_uint64)) for r in range(requests)]
    new_all = new.ctypes.data_as(C.POINTER(C.c_uint64))
    s_h = C.c_void_p(stream.cuda_stream)

    def once():
        for r in range(requests):
            st = lib.t2i_pull(cons._h, hw.store._h, src_p[r], n, 0, dst_p[r], None, s_h)
            if st:
                raise RuntimeError("pull: " + cons.last_error())
        cons.check(lib.t2i_free(cons._h, new_all, len(new)))

    once()
    torch.cuda.synchronize(device)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(reps):
        once()
    e1.record(stream)
    torch.cuda.synchronize(device)
    ms = e0.elapsed_time(e1) / reps

    # the same pulls with request r on stream r % 4 (independent requests overlap)
    streams = [stream] + [torch.cuda.Stream(device) for _ in range(3)]
    ss = [C.c_void_p(x.cuda_stream) for x in streams]

    def once4():
        for r in range(requests):
            st = lib.t2i_pull(cons._h, hw.store._h, src_p[r], n, 0, dst_p[r], None, ss[r % 4])
            if st:
                raise RuntimeError("pull: " + cons.last_error())
        cons.check(lib.t2i_free(cons._h, new_all, len(new)))

    once4()
    torch.cuda.synchronize(device)
    e0.record(stream)
    for x in streams[1:]:
        x.wait_event(e0)
    for _ in range(reps):
        once4()
    for x in streams[1:]:
        ev = torch.cuda.Event()
        ev.record(x)
        stream.wait_event(ev)
    e1.record(stream)
    torch.cuda.synchronize(device)
    ms4 = e0.elapsed_time(e1) / reps
    # the consumer's bytes equal the producer's (a sample request)
    from paper_2607_26566_gb300 import get_descs
    st, out, _ = cons.pull(hw.store, hw.ids[:n])
    cons.check(st)
    dst = [torch.empty(sp.nbytes, dtype=torch.uint8, device=device) for sp in hw.specs]
    cons.check(cons.get_batch(get_descs(out, dst), per_item=False)[0])
    torch.cuda.synchronize(device)
    ok = all(torch.equal(t.reshape(-1).view(torch.uint8), d) for t, d in zip(hw.inputs[0], dst))
    res = {"workload": f"pull: {requests} handoff requests (B={B}) from a producer store into a consumer store",
           "ms": round(ms, 3), "gbs": round(2 * payload / (ms * 1e-3) / 1e9, 1), "bit_exact": bool(ok),
           "streams4_ms": round(ms4, 3), "streams4_gbs": round(2 * payload / (ms4 * 1e-3) / 1e9, 1)}
    cons.close()
    hw.store.close()
    del hw, cons, cons_pool
    torch.cuda.empty_cache()
    return res


def _ipc_producer(to_parent, from_parent, B: int, requests: int, seed: int, device_index: int):
    """A producer executor in its own process: puts the handoff requests into
    its store and shares the pool (CUDA IPC, through torch) and the page
    lists with the consumer, until the consumer is done."""
    import torch

    from paper_2607_26566_gb300 import Store, put_descs

    dev = torch.device("cuda", device_index)
    torch.cuda.set_device(dev)
    specs = W.handoff_specs(B)
    pool = torch.empty(W.HANDOFF["pool_bytes"], dtype=torch.uint8, device=dev)
    st = Store(pool, W.HANDOFF["page_bytes"])
    objects = []
    for r in range(requests):
        ts = W.handoff_request_torch(seed, r, specs, dev)
        s, ids = st.put_batch(put_descs(ts, nbytes=[sp.nbytes for sp in specs]))
        st.check(s)
        objects.append([(sp.nbytes, st.ctl.object(int(i))[2], sp.dtype_tag) for sp, i in zip(specs, ids)])
        torch.cuda.synchronize(dev)
        del ts
    to_parent.put((pool, objects))
    from_parent.get(timeout=600)
    st.close()


def time_pull_ipc(device, B: int = 8, requests: int = 64, reps: int = 3, n_streams: int = 4, seed: int = 5):
    """The handoff pulled across processes: a spawned producer shares its
    store's pool through CUDA IPC, and this process pulls every request into
    its own store with t2i_pull_pages, request r on stream r % n_streams."""
    import torch
    import torch.multiprocessing as tmp

    from paper_2607_26566_gb300 import Store, get_descs
    from paper_2607_26566_gb300 import _lib as L

    ctx = tmp.get_context("spawn")
    to_parent, from_parent = ctx.Queue(), ctx.Queue()
    child = ctx.Process(target=_ipc_producer, args=(to_parent, from_parent, B, requests, seed, device.index or 0))
    child.start()
    try:
        src_pool, objects = to_parent.get(timeout=600)
        cons = Store(torch.empty(W.HANDOFF["pool_bytes"], dtype=torch.uint8, device=device), W.HANDOFF["page_bytes"])
        lib = cons._lib
        # C arrays built once: each pull is a raw C-ABI call
        keep, arrays = [], []
        for objs in objects:
            arr = (L.PagedObject * len(objs))()
            for j, (nb, pages, tag) in enumerate(objs):
                pg = np.ascontiguousarray(pages, np.uint32)
                keep.append(pg)
                arr[j] = L.PagedObject(int(nb), pg.ctypes.data, len(pg), int(tag))
            arrays.append(arr)
        n = len(objects[0])
        new = np.zeros(requests * n, np.uint64)
        streams = [torch.cuda.current_stream(device)] + [torch.cuda.Stream(device) for _ in range(n_streams - 1)]
        ss = [C.c_void_p(x.cuda_stream) for x in streams]
        sp, spb = src_pool.data_ptr(), src_pool.numel()

        def once():
            for r in range(requests):
                st = lib.t2i_pull_pages(cons._h, sp, spb, C.addressof(arrays[r]), n, 0,
                                        new.ctypes.data + 8 * n * r, ss[r % n_streams])
                if st:
                    raise RuntimeError("pull_pages: " + cons.last_error())
            cons.check(cons.free(new))

        once()
        torch.cuda.synchronize(device)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(streams[0])
        for x in streams[1:]:
            x.wait_event(e0)
        for _ in range(reps):
            once()
        for x in streams[1:]:
            ev = torch.cuda.Event()
            ev.record(x)
            streams[0].wait_event(ev)
        e1.record(streams[0])
        torch.cuda.synchronize(device)
        ms = e0.elapsed_time(e1) / reps
        payload = sum(nb for objs in objects for nb, _, _ in objs)
        # request 0 pulled once more and compared with its inputs
        s, ids = cons.pull_pages(src_pool, objects[0])
        cons.check(s)
        specs = W.handoff_specs(B)
        want = W.handoff_request_torch(seed, 0, specs, device)
        outs = [torch.empty(sp.nbytes, dtype=torch.uint8, device=device) for sp in specs]
        cons.check(cons.get_batch(get_descs(ids, outs), per_item=False)[0])
        torch.cuda.synchronize(device)
        ok = all(torch.equal(t.reshape(-1).view(torch.uint8), o) for t, o in zip(want, outs))
        res = {"ipc_workload": f"the {requests} B={B} requests pulled from a producer process's store (CUDA IPC), "
                               f"{n_streams} streams",
               "ipc_ms": round(ms, 3), "ipc_gbs": round(2 * payload / (ms * 1e-3) / 1e9, 1), "ipc_bit_exact": bool(ok)}
        cons.close()
        del src_pool
        from_parent.put("done")
        child.join(timeout=120)
        return res
    finally:
        if child.is_alive():
            child.terminate()
            child.join(timeout=30)


# ----------------------------------------------------------------------------- CPU (oracle)
def oracle_sample(B: int, n_requests: int, min_seconds: float = 0.0, max_steps: int = 1):
    """The oracle as it stands on the host: steps of the handoff workload (put
    all ``n_requests`` requests, get them with the latents cast, free them),
    repeated until ``min_seconds`` have passed or ``max_steps`` were run. The
    inputs of one request are reused for all requests (the oracle copies
    them). Returns (GB/s, seconds, bytes, steps)."""
    from oracle import OracleStore, PutItem

    specs = W.handoff_specs(B)
    arrs = W.handoff_request(0, 0, specs)
    raw = [a.view(np.uint8).reshape(-1) for a in arrs]
    ci = W.handoff_cast_index()
    casts = [1 if j == ci else 0 for j in range(len(specs))]
    store = OracleStore(W.HANDOFF["pool_bytes"], W.HANDOFF["page_bytes"])
    payload = sum(sp.nbytes for sp in specs)
    lat = specs[ci].nbytes
    per_req = 2 * payload + 2 * (payload - lat) + 1.5 * lat
    t = time.perf_counter()
    steps = 0
    while True:
        ids_all = []
        for _ in range(n_requests):
            st, ids = store.put_batch([PutItem(x.size, x, sp.dtype_tag) for x, sp in zip(raw, specs)])
            ids_all.append(ids)
        for ids in ids_all:
            store.get_batch(ids, casts)
        for ids in ids_all:
            store.free(ids)
        steps += 1
        dt = time.perf_counter() - t
        if steps >= max_steps and dt >= min_seconds:
            break
    return per_req * n_requests * steps / dt / 1e9, dt, per_req * n_requests * steps, steps


def host_memcpy_sample(B: int, n_requests: int, min_seconds: float = 2.0, threads: int | None = None):
    """A multithreaded host memcpy of the same step on the host cores: every
    request's objects copied into 2 MiB pages of a host pool (put), then out
    into consumer arrays (get, latents copied as fp32: no cast), split over
    ``threads`` threads (numpy copies release the GIL). A reported baseline,
    not the oracle. Returns (GB/s of 2 x copied bytes, seconds, threads)."""
    from concurrent.futures import ThreadPoolExecutor

    threads = threads or os.cpu_count() or 1
    specs = W.handoff_specs(B)
    P = W.HANDOFF["page_bytes"]
    src = [np.random.default_rng(j).integers(0, 256, sp.nbytes, dtype=np.uint8) for j, sp in enumerate(specs)]
    pages = sum(-(-sp.nbytes // P) for sp in specs)
    pool = np.empty(n_requests * pages * P, np.uint8)
    dst = [[np.empty(sp.nbytes, np.uint8) for sp in specs] for _ in range(n_requests)]
    put, get = [], []
    pg = 0
    for r in range(n_requests):
        for j, sp in enumerate(specs):
            for o in range(0, sp.nbytes, P):
                n = min(P, sp.nbytes - o)
                put.append((pool[pg * P:pg * P + n], src[j][o:o + n]))
                get.append((dst[r][j][o:o + n], pool[pg * P:pg * P + n]))
                pg += 1
    nbytes = 2 * sum(a.size for a, _ in put) * 2

    def part(lst, i):
        for a, b in lst[i::threads]:
            np.copyto(a, b)

    with ThreadPoolExecutor(threads) as ex:
        for phase in (put, get):          # warm-up: touch every page
            list(ex.map(lambda i: part(phase, i), range(threads)))
        t = time.perf_counter()
        steps = 0
        while True:
            for phase in (put, get):
                list(ex.map(lambda i: part(phase, i), range(threads)))
            steps += 1
            dt = time.perf_counter() - t
            if dt >= min_seconds:
                break
    return nbytes * steps / dt / 1e9, dt, threads


def oracle_row_samples(rows: dict) -> None:
    """The oracle as it stands, on a bounded sample of each row's workload
    (single thread, the same byte counting as the row), added to the row as
    ``cpu_oracle``. A reported baseline, not a target."""
    from oracle import OK, OracleStore, PutItem

    def entry(nbytes, dt, sample):
        return {"value": round(nbytes / dt / 1e9, 3), "unit": "GB/s", "cores": 1, "kind": "oracle",
                "sample": f"{sample}, {dt:.2f} s"}

    if "weights" in rows:
        specs = W.dit_weight_specs()
        blk = [i for i, sp in enumerate(specs) if sp.block == 0]
        g = np.random.default_rng(0)
        data = [g.integers(0, 256, specs[i].nbytes, dtype=np.uint8) for i in blk]
        ora = OracleStore(W.WEIGHTS["pool_bytes"], W.WEIGHTS["page_bytes"])
        t = time.perf_counter()
        st, ids = ora.put_batch([PutItem(d.size, d, W.DTYPE_BF16, 0, 0, True) for d in data])
        st2, _, outs = ora.get_batch(ids)
        dt = time.perf_counter() - t
        assert st == OK and st2 == OK
        n = sum(d.size for d in data)
        rows["weights"]["cpu_oracle"] = entry(4 * n, dt, f"put + get of block 0 ({len(blk)} tensors, "
                                                         f"{n / 2**20:.0f} MiB)")
    if "adapters" in rows:
        ranks = W.lora_ranks(0, 4)
        ora = OracleStore(W.ADAPTERS["pool_bytes"], W.ADAPTERS["page_bytes"])
        g = np.random.default_rng(0)
        sets = []
        for s_, r in enumerate(ranks):
            objs = W.lora_objects(int(r))
            st, ids = ora.put_batch([PutItem(nb, g.integers(0, 256, nb, dtype=np.uint8), W.DTYPE_BF16, s_, b, True)
                                     for b, nb in objs])
            assert st == OK
            sets.append((ids, [nb for _, nb in objs]))
        t = time.perf_counter()
        nbytes = 0
        for k in range(100):
            ids, sz = sets[k % len(sets)]
            w = (97 * k) % (len(ids) - 256)
            st, _, _ = ora.get_batch(ids[w:w + 256])
            assert st == OK
            nbytes += 2 * sum(sz[w:w + 256])
        rows["adapters"]["cpu_oracle"] = entry(nbytes, time.perf_counter() - t,
                                               "100 hit gets of 256 objects over 4 resident sets")
    if "compaction" in rows:
        C_ = W.COMPACTION
        pool = 4 << 30
        P = C_["page_bytes"]
        tr = W.compaction_trace(1, pool // P, P, 6250, C_["lo"], pool // 128, C_["p_free"], C_["settle_frac"])
        ora = OracleStore(pool, P, keep_bytes=False, paged_pool=True)
        ids = {}
        for op in tr.ops:
            if op[0] == "alloc":
                ids[op[1]] = ora.put_batch([PutItem(op[2])])[1][0]
            else:
                ora.free([ids.pop(op[1])])
        t = time.perf_counter()
        st, moves = ora.compact(pool * 3 // 4)
        dt = time.perf_counter() - t
        assert st == OK
        rows["compaction"]["cpu_oracle"] = entry(2 * sum(m[2] for m in moves), dt,
                                                 f"compact of a 4 GiB paged pool to 3/4 ({len(moves)} pages moved)")


# ----------------------------------------------------------------------------- host control
def time_host_control(reps: int = 200) -> dict:
    """The host steps of the path (§8 a1, a2, a7, a9) alone, through the
    store's control core (t2i_ctl_*: the same code every store runs before
    its launches), on the host: median µs per call."""
    from paper_2607_26566_gb300 import Ctl, get_descs, put_descs

    def med(fn, n):
        ts = []
        for _ in range(n):
            t = time.perf_counter()
            fn()
            ts.append(time.perf_counter() - t)
        return round(1e6 * statistics.median(ts), 2)

    out = {"workload": "host control core alone (t2i_ctl_*), median µs per call"}
    # a1 + a2 + a9: put and free of one B=8 handoff request (4 objects, 45 pages of 2 MiB)
    C_ = W.HANDOFF
    specs = W.handoff_specs(8)
    ctl = Ctl(C_["pool_bytes"] // C_["page_bytes"], C_["page_bytes"])
    pd = put_descs([0] * len(specs), nbytes=[sp.nbytes for sp in specs])
    ids = [None]

    def put():
        st, ids[0] = ctl.put(pd)
        assert st == 0

    def free():
        assert ctl.free(ids[0]) == 0

    put_t, free_t = [], []
    for _ in range(reps):
        t = time.perf_counter()
        put()
        put_t.append(time.perf_counter() - t)
        t = time.perf_counter()
        free()
        free_t.append(time.perf_counter() - t)
    out["handoff_put_us"] = round(1e6 * statistics.median(put_t), 2)
    out["handoff_free_us"] = round(1e6 * statistics.median(free_t), 2)
    put()
    gd = get_descs(ids[0])
    out["handoff_get_us"] = med(lambda: ctl.get(gd), reps)
    ctl.close()
    # a7: adapter sets (836 objects each, 256 KiB pages, 16 GiB pool); once
    # the pool is full every set put evicts the least recently used set
    A = W.ADAPTERS
    ctl = Ctl(A["pool_bytes"] // A["page_bytes"], A["page_bytes"])
    ranks = W.lora_ranks(0)
    sets = []
    for s_, r in enumerate(ranks[:64]):
        objs = W.lora_objects(int(r))
        sets.append(put_descs([0] * len(objs), nbytes=[nb for _, nb in objs], group=s_,
                              order=[b for b, _ in objs], evictable=1))
    put_t, evicted, live = [], 0, {}
    for k in range(3 * len(sets)):
        s_ = k % len(sets)
        t = time.perf_counter()
        st, got = ctl.put(sets[s_])
        put_t.append(time.perf_counter() - t)
        assert st == 0
        ev = ctl.last_evictions()
        evicted += len(ev)
        live[s_] = got
    steady = put_t[len(sets):]
    out["adapter_set_put_us"] = round(1e6 * statistics.median(steady), 2)
    out["adapter_set_put_evictions_per_call"] = round(evicted / len(put_t), 1)
    # the 256-object hit get of one resident window (validation + LRU stamps)
    last = (3 * len(sets) - 1) % len(sets)
    gd = get_descs(live[last][:256])
    out["adapter_get_256_us"] = med(lambda: ctl.get(gd), reps)
    ctl.close()
    # a8: compaction planning of the 64 GiB, 100,000-op fragmentation trace
    C5 = W.COMPACTION
    P = C5["page_bytes"]
    tr = W.compaction_trace(1, C5["pool_bytes"] // P, P, C5["n_ops"], C5["lo"], C5["hi"], C5["p_free"],
                            C5["settle_frac"])
    ctl = Ctl(C5["pool_bytes"] // P, P)
    oid = {}
    for op in tr.ops:
        if op[0] == "alloc":
            st, got = ctl.put(put_descs([0], nbytes=[op[2]]))
            assert st == 0
            oid[op[1]] = int(got[0])
        else:
            assert ctl.free([oid.pop(op[1])]) == 0
    t = time.perf_counter()
    st, moves = ctl.compact(C5["limit_bytes"])
    out["compaction_plan_ms"] = round(1e3 * (time.perf_counter() - t), 3)
    out["compaction_moves"] = int(len(moves)) if st == 0 else None
    ctl.close()
    out["note"] = "through the Python binding (ctypes, descriptor arrays built beforehand)"
    return out


# ----------------------------------------------------------------------------- main
def arm_config(args, world: int) -> dict:
    """The workload both arms name (the reference arm times a bounded sample
    of it, described in its ``cpu_baseline.sample``)."""
    pool_bytes = int(args.pool_gib * (1 << 30)) if args.pool_gib else None
    return {"workload": f"t2i handoff, B={args.batch}, {args.requests} requests in flight",
            "streams": args.streams,
            "pool_bytes": pool_bytes or W.HANDOFF["pool_bytes"], "page_bytes": W.HANDOFF["page_bytes"],
            "bytes_per_step": hw_bytes(args.batch, args.requests), "l2": "inputs > L2 (no flush)",
            "parallelism": f"replicas x{world}"}


def run_reference(args, dist_ctx):
    if dist_ctx.rank != 0:
        return
    B = args.batch
    n_req = 8   # a bounded sample of the 64 requests of one step
    for _ in range(args.warmup):
        oracle_sample(B, 1)
    vals = []
    t0 = time.perf_counter()
    nb = 0
    for _ in range(args.steps):
        v, dt, nb, _ = oracle_sample(B, n_req)
        vals.append((v, dt))
    total_t = sum(dt for _, dt in vals)
    total_b = sum(v * dt for v, dt in vals)
    value = total_b / total_t
    ms = 1e3 * total_t / len(vals)
    line = {
        "impl": "reference", "metric": METRIC, "value": round(value, 3), "unit": "GB/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 3), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "u8+f32->bf16", "data": "synthetic",
        "config": arm_config(args, dist_ctx.world),
        "cpu_baseline": {"value": round(value, 3), "unit": "GB/s", "cores": 1, "kind": "oracle",
                         "sample": f"each step: {n_req} of the step's {args.requests} B={B} requests (put, get with "
                                   f"the latents cast, free), numpy oracle, single thread"},
        "e2e": {"value": round(value, 3), "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        "sampled_bytes_per_step": int(nb),   # ms_per_step is the time of this sample
        "wall_s": round(time.perf_counter() - t0, 2),
    }
    print(json.dumps(line), flush=True)


def run_rows(args, device, peak):
    rows = {}
    wanted = [] if args.rows == "none" else [r.strip() for r in args.rows.split(",") if r.strip()]
    if "tiny" in wanted:
        rows["tiny"] = time_tiny(device)
    if "unaligned" in wanted:
        rows["unaligned"] = time_unaligned(device)
    if "cdriver" in wanted:
        rows["cdriver"] = time_c_driver(device)
    if "host" in wanted:
        rows["host"] = time_host_control()
    if "weights" in wanted:
        rows["weights"] = time_weights(device, n_blocks=args.weight_blocks)
    if "adapters" in wanted:
        rows["adapters"] = time_adapters(device, n_calls=args.adapter_calls, n_sets=args.adapter_sets,
                                         pool_bytes=int(args.adapter_pool_gib * (1 << 30)) if args.adapter_pool_gib
                                         else None)
    if "compaction" in wanted:
        rows["compaction"] = time_compaction(device, pool_gib=args.compaction_gib)
    if "prefix" in wanted:
        rows["prefix"] = time_prefix(device)
    if "views" in wanted:
        rows["views"] = time_views(device)
    if "pull" in wanted:
        rows["pull"] = time_pull(device)
        try:
            rows["pull"].update(time_pull_ipc(device))
        except Exception as e:  # a box without CUDA IPC: the same-process row stands
            rows["pull"]["ipc_error"] = f"{type(e).__name__}: {e}"
    for r in rows.values():
        for k in ("get_gbs", "gbs", "hit_gbs"):
            if k in r:
                r[k.replace("gbs", "hbm_frac")] = round(r[k] / peak, 4)
    return rows


def main():
    args = parse()
    # the reference arm runs on rank 0 alone and needs no process group
    dist_ctx = Dist(init=args.impl != "reference")
    if args.impl == "reference":
        run_reference(args, dist_ctx)
        dist_ctx.close()
        return
    import torch

    from paper_2607_26566_gb300 import build as b

    if args.lib:
        # a library built with other compile-time launch shapes (tuning
        # sweeps): every call goes to it through ctypes (the CPython module
        # is linked against the package's own library)
        from paper_2607_26566_gb300 import _lib as L

        if L._lib is not None:
            raise RuntimeError("--lib must be set before the library is loaded")
        L.LIB_PATH = os.path.abspath(args.lib)
        L._pycall = None
    else:
        b.ensure_built()
    device = torch.device("cuda", dist_ctx.local)
    torch.cuda.set_device(device)
    if args.rows_only:
        print(json.dumps({"rows": run_rows(args, device, peaks()[0])}), flush=True)
        dist_ctx.close()
        return
    B = args.batch
    pool_bytes = int(args.pool_gib * (1 << 30)) if args.pool_gib else None
    hw = Handoff(B, args.requests, device, pool_bytes=pool_bytes)
    ms, launches, kern, clocks = time_handoff(hw, args.steps, args.warmup, dist_ctx, per_kernel=True,
                                              clocks_index=dist_ctx.local, n_streams=args.streams)
    hw.verify()
    ms_max = dist_ctx.max(ms)
    value = job_gbs(hw.step_bytes * args.steps, ms_max, dist_ctx)
    peak, peak_kind = peaks()

    def rates(kn):
        return {"put": kn["put_phase_bytes"] / (kn["put_phase_ms"] * 1e-3) / 1e9,
                "get": kn["get_phase_bytes"] / (kn["get_phase_ms"] * 1e-3) / 1e9}

    # dominant kernel: the one with more time in the timed region; its phase
    # (hw.requests launches, args.streams at a time) moves phase_bytes
    dom = "gather_get_kernel" if kern["get_phase_ms"] >= kern["put_phase_ms"] else "scatter_put_kernel"
    d, o = ("get", "put") if dom == "gather_get_kernel" else ("put", "get")
    achieved = rates(kern)[d]
    traffic = ncu_traffic(dom, f"handoff_B{B}_request")
    roofline = {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                "frac": round(achieved / peak, 4), "peak_kind": peak_kind,
                "traffic": traffic,
                "kernel": dom, "algorithmic_bytes_per_launch": kern[f"{d}_phase_bytes"] / hw.requests,
                "launches_per_phase": hw.requests, "streams": args.streams,
                "phase_ms": round(kern[f"{d}_phase_ms"], 5),
                "achieved_is": "algorithmic bytes of the phase's launches / phase span (CUDA events)",
                "other_kernel": {"name": "scatter_put_kernel" if d == "get" else "gather_get_kernel",
                                 "achieved": round(rates(kern)[o], 1)}}
    if args.streams > 1:
        # the same workload on one stream: back-to-back launches, so the phase
        # span / launches is each launch's own duration
        ms1, _, kern1, _ = time_handoff(hw, max(3, args.steps // 2), args.warmup, dist_ctx, per_kernel=True,
                                        nvtx="bench_one_stream")
        r1 = rates(kern1)
        roofline["one_stream"] = {"step_gbs": round(job_gbs(hw.step_bytes * max(3, args.steps // 2), dist_ctx.max(ms1),
                                                            dist_ctx), 1),
                                  "get_achieved": round(r1["get"], 1), "put_achieved": round(r1["put"], 1),
                                  "get_frac": round(r1["get"] / peak, 4),
                                  "get_avg_launch_ms": round(kern1["get_phase_ms"] / hw.requests, 5)}
    per_call = time_calls(hw)
    del hw
    torch.cuda.empty_cache()

    # the same bytes in one call per phase, and with reclaim by consumer count
    extras = {}
    if not args.no_extras:
        hx = Handoff(B, args.requests, device, pool_bytes=pool_bytes)
        stream = torch.cuda.current_stream(device)
        for _ in range(3):
            hx.step_one_call()
        torch.cuda.synchronize(device)
        a, z = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(10):
            hx.step_one_call()
        z.record(stream)
        torch.cuda.synchronize(device)
        extras["one_call_per_phase_gbs"] = round(hx.step_bytes * 10 / (a.elapsed_time(z) * 1e-3) / 1e9, 1)
        hx.store.close()
        del hx
        hr = Handoff(B, args.requests, device, pool_bytes=pool_bytes, consumers=1)
        ms_r, _, _, _ = time_handoff(hr, 10, 3, dist_ctx, per_kernel=False, nvtx="bench_reclaim")
        extras["reclaim_by_consumers_gbs"] = round(hr.step_bytes * 10 / (ms_r * 1e-3) / 1e9, 1)
        extras["reclaimed_per_step"] = hr.store.stats()["reclaimed"] // 13
        hr.store.close()
        del hr
        torch.cuda.empty_cache()

    sweep = {}
    if not args.no_sweep:
        for Bs in (1, 4):
            hs = Handoff(Bs, args.requests, device)
            ms_s, _, _, _ = time_handoff(hs, max(3, args.steps // 2), args.warmup, dist_ctx, per_kernel=False,
                                         n_streams=args.streams, nvtx="bench_sweep")
            sweep[f"B{Bs}"] = round(hs.step_bytes * max(3, args.steps // 2) / (ms_s * 1e-3) / 1e9, 1)
            if Bs == 1:
                # small requests: the same on one stream, and one call per phase
                ms_1, _, _, _ = time_handoff(hs, max(3, args.steps // 2), args.warmup, dist_ctx, per_kernel=False,
                                             nvtx="bench_sweep")
                sweep["B1_one_stream"] = round(hs.step_bytes * max(3, args.steps // 2) / (ms_1 * 1e-3) / 1e9, 1)
                stream = torch.cuda.current_stream(device)
                for _ in range(3):
                    hs.step_one_call()
                torch.cuda.synchronize(device)
                a, z = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record(stream)
                for _ in range(10):
                    hs.step_one_call()
                z.record(stream)
                torch.cuda.synchronize(device)
                sweep["B1_one_call_per_phase"] = round(hs.step_bytes * 10 / (a.elapsed_time(z) * 1e-3) / 1e9, 1)
            del hs
            torch.cuda.empty_cache()

    e2e = None
    if not args.no_e2e:
        he = Handoff(B, args.requests, device, host_buffers=True)
        e_steps = max(2, min(args.steps, 10))
        # the kernels read and write host memory themselves (h2d_mode = d2h_mode = 0)
        ms_e, _, _, _ = time_handoff(he, e_steps, 3, dist_ctx, per_kernel=False, n_streams=args.streams,
                                     nvtx="bench_e2e")
        ms_e = dist_ctx.max(ms_e)
        ms_e1, _, _, _ = time_handoff(he, e_steps, 1, dist_ctx, per_kernel=False, nvtx="bench_e2e")
        ms_e1 = dist_ctx.max(ms_e1)
        ms_k2 = dist_ctx.max(time_two_streams(he, e_steps))
        he.verify()
        # the headline end-to-end form: host copies on the copy engines
        # (h2d_mode = d2h_mode = 1; the latents' cast stays in the kernel),
        # puts on one stream and gets on another, so that host-to-device and
        # device-to-host transfers overlap on the link
        he.reopen(h2d_mode=1, d2h_mode=1)
        ms_c2_lifo = dist_ctx.max(time_two_streams(he, e_steps))
        he.verify()
        # ... under extent placement: a step's first puts take the lowest free
        # pages, whose gets ended early in the step before, instead of the
        # pages of its last get (LIFO), so steps overlap on the link too
        he.reopen(h2d_mode=1, d2h_mode=1, alloc_policy=1)
        # three measurements, the median reported: the host link is shared with
        # the rest of the machine, and one measurement can land in a burst of
        # someone else's traffic
        ms_c2_reps = [dist_ctx.max(time_two_streams(he, e_steps)) for _ in range(3)]
        ms_c2 = statistics.median(ms_c2_reps)
        he.verify()
        gbs = lambda ms: round(job_gbs(he.step_bytes * e_steps, ms, dist_ctx), 2)  # noqa: E731
        e2e = {"value": gbs(ms_c2), "unit": "GB/s",
               "h2d_bytes_per_step": int(he.h2d_bytes), "d2h_bytes_per_step": int(he.d2h_bytes),
               "path": "t2i_put_batch / t2i_get_batch with pinned host sources and destinations; copy engines "
                       "for the host copies (h2d_mode = d2h_mode = 1), extent placement (alloc_policy = 1); "
                       "puts on one stream, gets on another",
               "link_gbs": round((he.h2d_bytes + he.d2h_bytes) * e_steps / (ms_c2 * 1e-3) / 1e9, 1),
               "measurements": [gbs(m) for m in ms_c2_reps],
               "lifo_placement_value": gbs(ms_c2_lifo),
               "kernel_host_copies": {"streams4_value": gbs(ms_e), "one_stream_value": gbs(ms_e1),
                                      "puts_and_gets_on_two_streams_value": gbs(ms_k2)}}
        del he
        torch.cuda.empty_cache()

    rows = run_rows(args, device, peak)
    if not args.no_cpu and dist_ctx.rank == 0:
        oracle_row_samples(rows)

    cpu = None
    if not args.no_cpu and dist_ctx.rank == 0:
        v, dt, nb, n = oracle_sample(B, args.requests, min_seconds=args.cpu_seconds, max_steps=1)
        cpu = {"value": round(v, 3), "unit": "GB/s", "cores": 1, "kind": "oracle",
               "sample": f"{n} full step(s) ({args.requests} B={B} requests put, got with the latents cast, "
                         f"freed) by the numpy oracle in {dt:.1f} s"}
        mv, mdt, mthreads = host_memcpy_sample(B, 8)
        cpu["host_memcpy"] = {"value": round(mv, 2), "unit": "GB/s", "cores": mthreads, "kind": "memcpy",
                              "sample": f"8 B={B} requests copied into 2 MiB pages of a host pool and out "
                                        f"again (no cast), {mthreads} threads, {mdt:.1f} s"}

    if dist_ctx.rank == 0:
        line = {
            "metric": METRIC, "value": round(value, 1), "unit": "GB/s", "n_gpus": dist_ctx.world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_max / args.steps, 4),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u8+f32->bf16",
            "data": "synthetic",
            "config": arm_config(args, dist_ctx.world),
            "hbm_frac": round(value / dist_ctx.world / peak, 4), "hbm_frac_nominal_8tbs": round(value / dist_ctx.world / 8000.0, 4),
            "step_ms": kern["step_ms"], "per_call": per_call,
            "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": int(launches),
            "clocks": clocks, "sweep": sweep or None, "extras": extras or None, "rows": rows or None,
        }
        print(json.dumps(line), flush=True)
    dist_ctx.close()


def hw_bytes(B, requests):
    specs = W.handoff_specs(B)
    payload = sum(sp.nbytes for sp in specs)
    lat = specs[W.handoff_cast_index()].nbytes
    return int((2 * payload + 2 * (payload - lat) + 1.5 * lat) * requests)


if __name__ == "__main__":
    main()
