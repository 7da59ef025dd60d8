"""Summarise an ncu launch list (``--metrics gpu__time_duration.sum --csv``) per kernel.

Usage: python -m paper_2607_14530_gb300.ncu_summary launches.csv [--last N]
Prints, per kernel, the number of launches, total device time and share of the total.  ``--last N``
keeps only the last N launches (one timed step after the warm-up steps).  The per-launch times
of such a list are cold-cache and serialised: compare shares, not absolute times.
"""
from __future__ import annotations

import csv
import io
import re
import sys


def load(path):
    with open(path) as f:
        text = f.read()
    start = text.find('"ID"')
    rows = list(csv.DictReader(io.StringIO(text[start:])))
    out = []
    for r in rows:
        if r.get("Metric Name") != "gpu__time_duration.sum":
            continue
        name = r["Kernel Name"]
        name = re.sub(r"\(.*$", "", name).replace("void ", "").strip()
        v = float(r["Metric Value"].replace(",", ""))
        unit = r.get("Metric Unit", "ns")
        scale = {"ns": 1e-6, "us": 1e-3, "usecond": 1e-3, "ms": 1.0, "msecond": 1.0, "nsecond": 1e-6}.get(unit, 1e-6)
        out.append((name, v * scale))
    return out


def summarise(launches):
    per = {}
    for n, ms in launches:
        e = per.setdefault(n, [0, 0.0])
        e[0] += 1
        e[1] += ms
    tot = sum(v[1] for v in per.values())
    lines = [f"{'kernel':28s} {'launches':>8s} {'total ms':>10s} {'share':>7s}"]
    for n, (c, t) in sorted(per.items(), key=lambda kv: -kv[1][1]):
        lines.append(f"{n:28s} {c:8d} {t:10.3f} {100 * t / tot:6.1f}%")
    lines.append(f"{'total':28s} {sum(v[0] for v in per.values()):8d} {tot:10.3f}")
    return "\n".join(lines)


if __name__ == "__main__":
    launches = load(sys.argv[1])
    if "--last" in sys.argv:
        launches = launches[-int(sys.argv[sys.argv.index("--last") + 1]):]
    print(summarise(launches))
