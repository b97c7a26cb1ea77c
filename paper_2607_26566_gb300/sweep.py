"""Tuning sweeps of the kernels' compile-time launch shapes (GPU).

Each variant is the library built with some ``T2I_TUNE_*`` definitions
(``csrc/kernels.cuh``, ``csrc/launch.cuh``, ``csrc/store.cu``); every variant
is timed by ``bench.py --lib`` in the same process order, alternating, for a
few repetitions, and one table line per run shows the figures the choices in
the kernels' comments were made on.

    python -m paper_2607_26566_gb300.sweep base= pf24=T2I_TUNE_PREFETCH_BYTES=24576 \\
        --bench "--no-e2e --no-cpu --rows adapters --adapter-calls 2000 --steps 30" --reps 2

A variant is ``NAME=DEF[,DEF...]`` (``NAME=`` alone: the defaults). Builds go
to ``_build/variants/``; the package's own library is not touched.
"""
from __future__ import annotations

import argparse
import json
import os
import shlex
import subprocess
import sys

from . import build as b

ROOT = os.path.dirname(b.PKG)
OUT = os.path.join(b.BUILD, "variants")


def build_variant(name: str, defines: list[str]) -> str:
    lib = os.path.join(OUT, f"libt2istore_{name}.so")
    b.build(defines=defines, out=lib, build_dir=os.path.join(OUT, f"_b_{name}"))
    return lib


def summary(line: dict) -> dict:
    """The figures of one bench line that the sweeps compare."""
    out = {"headline": line.get("value")}
    ro = line.get("roofline") or {}
    if ro:
        put = ro["achieved"] if ro.get("kernel") == "scatter_put_kernel" else ro.get("other_kernel", {}).get("achieved")
        get = ro["achieved"] if ro.get("kernel") == "gather_get_kernel" else ro.get("other_kernel", {}).get("achieved")
        out.update({"put_4s": put, "get_4s": get})
        one = ro.get("one_stream") or {}
        out.update({"step_1s": one.get("step_gbs"), "put_1s": one.get("put_achieved"),
                    "get_1s": one.get("get_achieved")})
    sw = line.get("sweep") or {}
    out.update({k: sw.get(k) for k in ("B1", "B1_one_stream", "B4")})
    rows = line.get("rows") or {}
    if "adapters" in rows:
        out["adapter_hits"] = rows["adapters"].get("hit_gbs")
    if "weights" in rows:
        out["weights_get"] = rows["weights"].get("get_gbs")
    if "compaction" in rows:
        out["compaction"] = rows["compaction"].get("gbs")
        out["compaction_call"] = rows["compaction"].get("call_gbs")
    if "unaligned" in rows:
        out.update({k: v for k, v in rows["unaligned"].items() if k.endswith("_gbs")})
    return {k: v for k, v in out.items() if v is not None}


def main(argv=None) -> int:
    p = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    p.add_argument("variants", nargs="+", help="NAME=DEF[,DEF...]")
    p.add_argument("--bench", default="--no-e2e --no-cpu --rows none --steps 30", help="bench.py arguments")
    p.add_argument("--reps", type=int, default=2)
    a = p.parse_args(argv)
    libs = {}
    for v in a.variants:
        name, _, defs = v.partition("=")
        libs[name] = build_variant(name, [d for d in defs.split(",") if d])
    for rep in range(a.reps):
        for name, lib in libs.items():
            cmd = [sys.executable, os.path.join(ROOT, "bench.py"), "--lib", lib] + shlex.split(a.bench)
            r = subprocess.run(cmd, capture_output=True, text=True, cwd=ROOT)
            if r.returncode:
                sys.stderr.write(r.stderr[-2000:])
                return r.returncode
            line = json.loads(r.stdout.strip().splitlines()[-1])
            if "rows" in line and "value" not in line:  # --rows-only
                line = {"rows": line["rows"]}
            print(json.dumps({"variant": name, "rep": rep, **summary(line)}), flush=True)
    return 0


if __name__ == "__main__":
    sys.exit(main())
