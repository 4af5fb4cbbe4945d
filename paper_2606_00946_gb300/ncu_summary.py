"""Summaries of ncu output for the profiles folder (text tables).

  python -m paper_2606_00946_gb300.ncu_summary launches <launches.csv>
      per kernel: launches, total device time and share of a
      `--metrics gpu__time_duration.sum --csv --log-file` run;
  python -m paper_2606_00946_gb300.ncu_summary full <report.ncu-rep>
      per captured launch: time, DRAM bytes, throughput and pipe
      utilisation, occupancy, registers, the three largest stall reasons.
"""
from __future__ import annotations

import csv
import subprocess
import sys
from collections import defaultdict


def _name(n: str) -> str:
    n = n.split("(")[0].replace("void ", "")
    for p in ("ls::", "(anonymous namespace)::", "<unnamed>::", "unnamed>::"):
        n = n.replace(p, "")
    return n


def launches(path: str) -> str:
    rows = list(csv.reader(open(path)))
    hdr, out = None, []
    for r in rows:
        if r and r[0] == "ID":
            hdr = r
            continue
        if hdr and len(r) == len(hdr):
            out.append(dict(zip(hdr, r)))
    agg = defaultdict(lambda: [0, 0.0, ""])
    for d in out:
        a = agg[_name(d["Kernel Name"])]
        a[0] += 1
        a[1] += float(d["Metric Value"]) / 1e3
        a[2] = d["Grid Size"]
    tot = sum(v[1] for v in agg.values())
    lines = ["| kernel | launches | total us | share | grid |", "|---|---|---|---|---|"]
    for k, v in sorted(agg.items(), key=lambda kv: -kv[1][1]):
        lines.append(f"| {k} | {v[0]} | {v[1]:.2f} | {100 * v[1] / tot:.1f}% | {v[2]} |")
    lines.append(f"| total | {len(out)} | {tot:.2f} | 100% | |")
    return "\n".join(lines)


COLS = [("time us", "gpu__time_duration.sum"), ("DRAM rd MB", "dram__bytes_read.sum"),
        ("DRAM wr MB", "dram__bytes_write.sum"), ("DRAM %", "gpu__dram_throughput.avg.pct_of_peak_sustained_elapsed"),
        ("SM %", "sm__throughput.avg.pct_of_peak_sustained_elapsed"),
        ("tensor %", "sm__pipe_tensor_cycles_active.avg.pct_of_peak_sustained_elapsed"),
        ("warps active %", "sm__warps_active.avg.pct_of_peak_sustained_active"),
        ("issue %", "smsp__issue_active.avg.pct_of_peak_sustained_active"), ("regs", "launch__registers_per_thread")]
SCALE = {"byte": 1e-6, "Kbyte": 1e-3, "Mbyte": 1.0, "Gbyte": 1e3, "nsecond": 1e-3, "usecond": 1.0, "msecond": 1e3}


def full(path: str) -> str:
    out = subprocess.run(["ncu", "-i", path, "--page", "raw", "--csv"], capture_output=True, text=True).stdout
    rows = list(csv.reader(out.splitlines()))
    hdr, units = rows[0], rows[1]
    lines = ["| # | kernel | grid x block | " + " | ".join(c for c, _ in COLS) + " | top stalls (per issue) |",
             "|---|---|---|" + "---|" * len(COLS) + "---|"]
    for k, r in enumerate(rows[2:]):
        vals = []
        for c, m in COLS:
            if m not in hdr:
                vals.append("n/a")
                continue
            i = hdr.index(m)
            try:
                f = float(r[i]) * (SCALE.get(units[i], 1.0) if c != "regs" and "%" not in c else 1.0)
                vals.append(str(int(f)) if c == "regs" else f"{f:.2f}")
            except ValueError:
                vals.append(r[i])
        st = [(hdr[i].replace("smsp__average_warps_issue_stalled_", "").replace("_per_issue_active.ratio", ""),
               float(r[i])) for i in range(len(hdr))
              if hdr[i].startswith("smsp__average_warps_issue_stalled_") and hdr[i].endswith("per_issue_active.ratio")
              and r[i]]
        st = ", ".join(f"{n} {v:.1f}" for n, v in sorted(st, key=lambda x: -x[1])[:3])
        grid = r[hdr.index("Grid Size")] + " x " + r[hdr.index("Block Size")]
        lines.append(f"| {k} | {_name(r[hdr.index('Kernel Name')])} | {grid} | " + " | ".join(vals) + f" | {st} |")
    return "\n".join(lines)


if __name__ == "__main__":
    mode, path = sys.argv[1], sys.argv[2]
    print(launches(path) if mode == "launches" else full(path))
