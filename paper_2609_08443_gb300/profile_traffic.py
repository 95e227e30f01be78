"""DRAM traffic of the tensor-core kernels, from an `ncu` capture of
`profile_case`, scaled to one call at the full workload size.

    python -m paper_2609_08443_gb300.profile_traffic prof.ncu-rep [more.ncu-rep ...] --config 4 --users 4 \
        > profiles/traffic.json

The capture runs a sub-batch of `--users` users with the workload's per-user
shapes; K/V streaming dominates the traffic and grows with the number of
tokens, so the bytes of each kernel are multiplied by (workload tokens /
sub-batch tokens).  bench.py reads the file and reports the traffic only while
`source_hash` matches the kernel sources it was built from.
"""
from __future__ import annotations

import argparse
import csv
import io
import json
import subprocess
import sys

from . import build, workloads as wl

_UNITS = {"byte": 1.0, "Kbyte": 1e3, "Mbyte": 1e6, "Gbyte": 1e9, "Tbyte": 1e12}


def kernel_bytes(report: str) -> dict:
    """Sum of dram__bytes_read.sum + dram__bytes_write.sum per kernel name
    (template arguments kept, parameter list dropped), with launch counts."""
    out = subprocess.run(["ncu", "-i", report, "--page", "raw", "--csv"], check=True, capture_output=True,
                         text=True).stdout
    rows = list(csv.reader(io.StringIO(out)))
    hdr, units = rows[0], rows[1]
    i_name = hdr.index("Kernel Name")
    cols = [hdr.index("dram__bytes_read.sum"), hdr.index("dram__bytes_write.sum")]
    agg = {}
    for r in rows[2:]:
        if len(r) <= max(cols):
            continue
        name = r[i_name].split("(")[0].replace("void ", "").split("::")[-1].replace(" ", "")
        if name.startswith("tc_fwd_kernel<"):  # the library names the forward's mode
            name = name[: name.rfind(",") + 1] + {"0>": "fused>", "1>": "sliced>", "2>": "pair>"}.get(name[name.rfind(",") + 1:], "?>")
        b = sum(float(r[c].replace(",", "")) * _UNITS[units[c]] for c in cols)
        e = agg.setdefault(name, {"bytes": 0.0, "launches": 0})
        e["bytes"] += b
        e["launches"] += 1
    return agg


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("report", nargs="+", help="ncu reports of profile_case on the same sub-batch")
    ap.add_argument("--config", type=int, default=4)
    ap.add_argument("--users", type=int, default=4)
    args = ap.parse_args()
    spec = wl.config(args.config)
    lens = wl.lengths(spec)
    scale = float(sum(lens)) / float(sum(lens[: args.users]))
    agg = {}
    for rep in args.report:
        agg.update(kernel_bytes(rep))
    h = build.source_hash()
    res = {}
    for name, e in sorted(agg.items()):
        res[name] = {"bytes_per_launch": e["bytes"] / e["launches"] * scale, "captured_launches": e["launches"],
                     "scale": scale, "source_hash": h}
    # the backward's two main kernels count as one call, as the bench times them
    for tok_pre, dq_pre in (("tc_bwd_tok_kernel", "tc_bwd_dq_kernel"), ("tc_tw_bwd_tok_kernel", "tc_tw_bwd_dq_kernel")):
        tok = next((k for k in res if k.startswith(tok_pre)), None)
        dq = next((k for k in res if k.startswith(dq_pre)), None)
        if tok and dq:
            res[tok]["bytes_per_call"] = res[tok]["bytes_per_launch"] + res[dq]["bytes_per_launch"]
    for name in res:
        res[name].setdefault("bytes_per_call", res[name]["bytes_per_launch"])
    json.dump(res, sys.stdout, indent=1, sort_keys=True)
    sys.stdout.write("\n")


if __name__ == "__main__":
    main()
