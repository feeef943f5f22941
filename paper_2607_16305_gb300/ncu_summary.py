"""Write a short Markdown summary of ncu output for profiles/.

  launches:  python -m paper_2607_16305_gb300.ncu_summary launches <launches.csv> <out.md> "<command>"
  kernel:    python -m paper_2607_16305_gb300.ncu_summary kernel <report.ncu-rep> <out.md> "<command>" <source.cu> <algorithmic_bytes>

The kernel summary records DRAM bytes per launch (traffic), throughput, warp
stall samples and the SHA-256 prefix of the kernel source it was taken on, so
that bench.py reports the traffic only while the kernel is unchanged.
"""
import collections
import csv
import hashlib
import io
import subprocess
import sys


def launches(csv_path, out, cmd):
    rows = list(csv.reader(open(csv_path)))
    hdr = None
    per = collections.defaultdict(list)
    for r in rows:
        if r and r[0] == "ID":
            hdr = r
            continue
        if hdr and len(r) == len(hdr):
            x = dict(zip(hdr, r))
            if x["Metric Name"] != "gpu__time_duration.sum":
                continue
            v = float(x["Metric Value"].replace(",", ""))
            unit = x["Metric Unit"]
            us = v / 1000.0 if unit in ("nsecond", "ns") else v * 1000.0 if unit in ("msecond", "ms") else v
            per[x["Kernel Name"].split("(")[0].replace("void ", "")].append(us)
    total = sum(sum(v) for k, v in per.items() if "lookme" in k)
    lines = [f"# ncu launch list: {out.split('/')[-1]}", "", "Command (run on one GB300):", "",
             f"    {cmd}", "",
             "Per-launch times are cold-cache and serialised (ncu); compare shares, not absolutes.", "",
             "| kernel | launches | total us | mean us | share of library time |", "|---|---|---|---|---|"]
    for k, v in sorted(per.items(), key=lambda kv: -sum(kv[1])):
        if "lookme" not in k:
            continue
        lines.append(f"| `{k}` | {len(v)} | {sum(v):.1f} | {sum(v) / len(v):.2f} | {100 * sum(v) / total:.1f}% |")
    open(out, "w").write("\n".join(lines) + "\n")


def kernel(rep, out, cmd, src, alg_bytes):
    raw = subprocess.run(["ncu", "-i", rep, "--page", "raw", "--csv"], capture_output=True, text=True).stdout
    rows = list(csv.reader(io.StringIO(raw)))
    hdr, units, vals = rows[0], rows[1], rows[2]
    get = {h: (vals[i], units[i]) for i, h in enumerate(hdr)}

    def num(name):
        v, u = get[name]
        v = float(v.replace(",", ""))
        scale = {"byte": 1, "Kbyte": 1e3, "Mbyte": 1e6, "Gbyte": 1e9, "nsecond": 1e-9, "usecond": 1e-6, "ns": 1e-9, "us": 1e-6, "ms": 1e-3,
                 "msecond": 1e-3}.get(u, 1)
        return v * scale

    name = get.get("Kernel Name", ("?", ""))[0]
    dur = num("gpu__time_duration.sum")
    rd, wr = num("dram__bytes_read.sum"), num("dram__bytes_write.sum")
    sha = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
    metrics = ["gpu__dram_throughput.avg.pct_of_peak_sustained_elapsed",
               "sm__pipe_tensor_cycles_active.avg.pct_of_peak_sustained_elapsed",
               "smsp__issue_active.avg.pct_of_peak_sustained_active",
               "sm__warps_active.avg.pct_of_peak_sustained_active", "launch__registers_per_thread",
               "launch__grid_size", "launch__block_size", "launch__shared_mem_per_block_dynamic"]
    stalls = sorted(((float(get[h][0].replace(",", "")), h) for h in get
                     if h.startswith("smsp__pcsamp_warps_issue_stalled") and not h.endswith("not_issued")
                     and get[h][0].replace(",", "").replace(".", "").isdigit()), reverse=True)[:6]
    lines = [f"# ncu --set full: {name}", "", "Command (run on one GB300):", "", f"    {cmd}", "",
             f"source_sha: {sha}", f"traffic_bytes_per_launch: {rd + wr:.0f}", "",
             "| quantity | value |", "|---|---|",
             f"| duration (ncu, cold L2, clocks uncontrolled) | {dur * 1e6:.2f} us |",
             f"| DRAM read | {rd / 1e6:.2f} MB |", f"| DRAM write | {wr / 1e6:.2f} MB |",
             f"| algorithmic bytes | {alg_bytes / 1e6:.2f} MB |",
             f"| traffic / algorithmic | {(rd + wr) / alg_bytes:.3f} |",
             f"| DRAM bandwidth over the launch | {(rd + wr) / dur / 1e9:.0f} GB/s |"]
    for m in metrics:
        if m in get:
            lines.append(f"| `{m}` | {get[m][0]} {get[m][1]} |")
    lines += ["", "Top warp-stall samples:", ""] + [f"- `{h}`: {v:.0f}" for v, h in stalls]
    open(out, "w").write("\n".join(lines) + "\n")


if __name__ == "__main__":
    if sys.argv[1] == "launches":
        launches(sys.argv[2], sys.argv[3], sys.argv[4])
    else:
        kernel(sys.argv[2], sys.argv[3], sys.argv[4], sys.argv[5], float(sys.argv[6]))
