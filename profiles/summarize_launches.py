"""Summarise an ncu launch-list CSV (gpu__time_duration.sum per launch) into
per-kernel launch counts, total time and share.  Usage:
  python profiles/summarize_launches.py launches.csv [--skip-prefix at::]"""
import csv
import sys
from collections import defaultdict


def main(path):
    rows = list(csv.reader(open(path)))
    hdr = None
    tot = defaultdict(float)
    cnt = defaultdict(int)
    for r in rows:
        if "Kernel Name" in r and "Metric Value" in r:
            hdr = r
            continue
        if hdr is None or len(r) != len(hdr):
            continue
        d = dict(zip(hdr, r))
        if d.get("Metric Name") != "gpu__time_duration.sum":
            continue
        name = d["Kernel Name"].split("(")[0]
        val = float(d["Metric Value"].replace(",", ""))
        unit = d.get("Metric Unit", "ns")
        scale = {"ns": 1e-3, "usecond": 1.0, "us": 1.0, "msecond": 1e3, "ms": 1e3, "nsecond": 1e-3}.get(unit, 1e-3)
        tot[name] += val * scale
        cnt[name] += 1
    total = sum(tot.values())
    print(f"{'kernel':60s} {'launches':>8s} {'total_us':>12s} {'share':>7s}")
    for name, t in sorted(tot.items(), key=lambda x: -x[1]):
        print(f"{name[:60]:60s} {cnt[name]:8d} {t:12.1f} {100 * t / total:6.1f}%")
    print(f"{'all':60s} {sum(cnt.values()):8d} {total:12.1f}")


if __name__ == "__main__":
    main(sys.argv[1])
