"""Summarise an Nsight Compute capture of the fused kernel for profiles/.

  python -m paper_2609_32479_gb300.ncu_summary full <raw.csv> <tracks> <out.md> <traffic.json> <cmd>
  python -m paper_2609_32479_gb300.ncu_summary launches <launches.csv> <out.md> <cmd>

`raw.csv` is `ncu -i <rep> --page raw --csv` of one captured launch; the
traffic JSON carries the DRAM bytes of that launch scaled to the full large
batch (1,048,576 tracks) and the sha256 of the kernel source it was taken on."""
from __future__ import annotations

import csv
import hashlib
import json
import os
import re
import sys
from collections import defaultdict

PKG = os.path.dirname(os.path.abspath(__file__))
KERNEL_SRC = os.path.join(PKG, "csrc", "tc_forward.cu")

KEYS = [
    ("gpu__time_duration.sum", "duration"),
    ("dram__bytes_read.sum", "DRAM read"),
    ("dram__bytes_write.sum", "DRAM write"),
    ("sm__pipe_tensor_cycles_active.avg.pct_of_peak_sustained_elapsed", "tensor pipe active"),
    ("smsp__issue_active.avg.pct_of_peak_sustained_active", "issue active"),
    ("sm__pipe_xu_cycles_active.avg.pct_of_peak_sustained_elapsed", "XU (MUFU) pipe active"),
    ("sm__pipe_fma_cycles_active.avg.pct_of_peak_sustained_elapsed", "FMA pipe active"),
    ("sm__pipe_alu_cycles_active.avg.pct_of_peak_sustained_elapsed", "ALU pipe active"),
    ("lts__throughput.avg.pct_of_peak_sustained_elapsed", "L2 throughput"),
    ("l1tex__m_xbar2l1tex_read_bytes_mem_global_op_tma_ld.sum", "TMA bytes L2->SM"),
    ("l1tex__m_xbar2l1tex_read_bytes_mem_global_op_tma_ld.sum.per_second", "TMA L2->SM rate"),
    ("gpu__dram_throughput.avg.pct_of_peak_sustained_elapsed", "DRAM throughput"),
    ("launch__registers_per_thread", "registers/thread"),
    ("smsp__average_warps_issue_stalled_long_scoreboard_per_issue_active.ratio", "stall long_scoreboard / issue"),
    ("smsp__average_warps_issue_stalled_wait_per_issue_active.ratio", "stall wait / issue"),
    ("smsp__average_warps_issue_stalled_short_scoreboard_per_issue_active.ratio", "stall short_scoreboard / issue"),
    ("smsp__average_warps_issue_stalled_branch_resolving_per_issue_active.ratio", "stall branch_resolving / issue"),
    ("smsp__average_warps_issue_stalled_barrier_per_issue_active.ratio", "stall barrier / issue"),
]

SCALE = {"byte": 1, "Kbyte": 1e3, "Mbyte": 1e6, "Gbyte": 1e9, "Tbyte": 1e12}


def _bytes(v, unit):
    return float(v.replace(",", "")) * SCALE.get(unit, 1.0)


def full(raw, tracks, out_md, out_json, cmd):
    rows = list(csv.reader(open(raw)))
    hdr, units, vals = rows[0], rows[1], rows[2]
    d = dict(zip(hdr, vals))
    u = dict(zip(hdr, units))
    how = "ncu --set full" if "--set full" in cmd else "ncu, the metrics below"
    lines = [f"# tc_forward_kernel, large workload ({tracks} tracks) — {how}", "",
             f"Command: `{cmd}`", "", "| metric | value |", "|---|---|"]
    for k, name in KEYS:
        if k in d:
            lines.append(f"| {name} (`{k}`) | {d[k]} {u[k]} |")
    rd = _bytes(d["dram__bytes_read.sum"], u["dram__bytes_read.sum"])
    wr = _bytes(d["dram__bytes_write.sum"], u["dram__bytes_write.sum"])
    per_track = (rd + wr) / tracks
    full_traffic = per_track * 1048576
    lines += ["", f"DRAM bytes per track: {per_track:.1f} (compulsory: 504); scaled to one 1,048,576-track "
                  f"launch: {full_traffic / 1e6:.1f} MB (traffic grows in proportion to the tracks)."]
    open(out_md, "w").write("\n".join(lines) + "\n")
    h = hashlib.sha256(open(KERNEL_SRC, "rb").read()).hexdigest()
    json.dump({"kernel": "tc_forward_kernel", "captured_tracks": tracks, "dram_bytes_captured": rd + wr,
               "dram_bytes_per_launch_full": full_traffic, "kernel_sha256": h, "command": cmd}, open(out_json, "w"),
              indent=1)


def launches(path, out_md, cmd):
    rows = [r for r in csv.reader(open(path)) if len(r) > 10]
    hdr = rows[0]
    ki, vi, ui = hdr.index("Kernel Name"), hdr.index("Metric Value"), hdr.index("Metric Unit")
    tot = defaultdict(float)
    cnt = defaultdict(int)
    for r in rows[1:]:
        name = re.sub(r"\(.*", "", r[ki]).split("::")[-1]
        scale = {"ns": 1e-6, "us": 1e-3, "ms": 1.0, "s": 1e3}.get(r[ui], 1e-6)
        tot[name] += float(r[vi].replace(",", "")) * scale
        cnt[name] += 1
    all_ms = sum(tot.values())
    lines = ["# Launch list of the bench command (ncu, gpu__time_duration.sum, cold and serialised)", "",
             f"Command: `{cmd}`", "", "| kernel | launches | total ms | share |", "|---|---|---|---|"]
    for n in sorted(tot, key=tot.get, reverse=True):
        lines.append(f"| {n} | {cnt[n]} | {tot[n]:.3f} | {100 * tot[n] / all_ms:.1f} % |")
    open(out_md, "w").write("\n".join(lines) + "\n")


if __name__ == "__main__":
    if sys.argv[1] == "full":
        full(sys.argv[2], int(sys.argv[3]), sys.argv[4], sys.argv[5], sys.argv[6])
    else:
        launches(sys.argv[2], sys.argv[3], sys.argv[4])
