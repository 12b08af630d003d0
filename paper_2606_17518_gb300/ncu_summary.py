"""Summaries of Nsight Compute output for the profiles kept with the library.

    python -m paper_2606_17518_gb300.ncu_summary launches LAUNCHES.csv
    python -m paper_2606_17518_gb300.ncu_summary report REPORT.ncu-rep

``launches``: a ``--metrics gpu__time_duration.sum --csv`` launch list, grouped
per kernel (launches, total device time, share).  Times from such a list are
cold-cache and serialised, so only the shares are comparable with the times a
benchmark measures.  ``report``: the memory, tensor-pipe and stall figures of
every launch in a ``--set full`` report (read with ``ncu -i ... --page raw``).
"""

from __future__ import annotations

import collections
import csv
import io
import re
import subprocess
import sys

_SCALE_US = {"ns": 1e-3, "nsecond": 1e-3, "us": 1.0, "usecond": 1.0, "ms": 1e3, "msecond": 1e3}

REPORT_METRICS = [
    "gpu__time_duration.sum",
    "dram__bytes_read.sum",
    "dram__bytes_write.sum",
    "gpu__dram_throughput.avg.pct_of_peak_sustained_elapsed",
    "sm__pipe_tensor_cycles_active.avg.pct_of_peak_sustained_elapsed",
    "sm__throughput.avg.pct_of_peak_sustained_elapsed",
    "sm__warps_active.avg.pct_of_peak_sustained_active",
    "lts__t_sector_hit_rate.pct",
    "launch__registers_per_thread",
    "launch__grid_size",
    "launch__block_size",
    "launch__shared_mem_per_block_dynamic",
]


def kernel_name(full: str) -> str:
    """Short kernel name: the function identifier without namespaces or arguments."""
    head = full.split("(")[0].replace("void ", "")
    while re.search(r"<[^<>]*>", head):  # template arguments (and "<unnamed>"), innermost first
        head = re.sub(r"<[^<>]*>", "", head)
    return head.split("::")[-1].strip()


def launches(path: str) -> str:
    rows = list(csv.reader(open(path, newline="")))
    hi = next(i for i, r in enumerate(rows) if "Kernel Name" in r)
    hdr = rows[hi]
    k, m, u, v = (hdr.index(x) for x in ("Kernel Name", "Metric Name", "Metric Unit", "Metric Value"))
    agg = collections.OrderedDict()
    for r in rows[hi + 1:]:
        if len(r) <= v or r[m] != "gpu__time_duration.sum":
            continue
        t = float(r[v].replace(",", "")) * _SCALE_US[r[u]]
        a = agg.setdefault(kernel_name(r[k]), [0, 0.0])
        a[0] += 1
        a[1] += t
    total = sum(t for _, t in agg.values()) or 1.0
    out = ["| kernel | launches | total us | share | mean us |", "|---|---:|---:|---:|---:|"]
    for name, (n, t) in sorted(agg.items(), key=lambda x: -x[1][1]):
        out.append(f"| {name} | {n} | {t:.1f} | {100 * t / total:.1f}% | {t / n:.2f} |")
    return "\n".join(out)


def report(path: str) -> str:
    raw = subprocess.run(["ncu", "-i", path, "--page", "raw", "--csv"], capture_output=True,
                         text=True, check=True).stdout
    rows = list(csv.reader(io.StringIO(raw)))
    hdr, units = rows[0], rows[1]
    out = []
    for vals in rows[2:]:
        name = kernel_name(vals[hdr.index("Kernel Name")]) if "Kernel Name" in hdr else "?"
        out.append(f"### {name}")
        out.append("| metric | value | unit |")
        out.append("|---|---:|---|")
        for mname in REPORT_METRICS:
            if mname in hdr:
                i = hdr.index(mname)
                out.append(f"| {mname} | {vals[i]} | {units[i]} |")
        stalls = []
        for i, h in enumerate(hdr):
            if h.startswith("smsp__average_warps_issue_stalled_") and h.endswith(
                    "_per_issue_active.ratio"):
                try:
                    stalls.append((float(vals[i]), h))
                except ValueError:
                    pass
        out.append("")
        out.append("top warp stalls (per issued instruction):")
        for val, h in sorted(stalls, reverse=True)[:6]:
            short = h[len("smsp__average_warps_issue_stalled_"):-len("_per_issue_active.ratio")]
            out.append(f"- {short}: {val:.2f}")
    return "\n".join(out)


if __name__ == "__main__":
    if len(sys.argv) != 3 or sys.argv[1] not in ("launches", "report"):
        raise SystemExit(__doc__)
    print(launches(sys.argv[2]) if sys.argv[1] == "launches" else report(sys.argv[2]))
