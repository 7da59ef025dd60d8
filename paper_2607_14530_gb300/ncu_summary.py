"""Summaries of ncu CSV logs.

Launch list (``--metrics gpu__time_duration.sum --csv``)::

    python -m paper_2607_14530_gb300.ncu_summary launches.csv [--last N]

prints, per kernel, the number of launches, total device time and share of the total.  ``--last
N`` keeps only the last N launches (one timed step after the warm-up steps).  The per-launch
times of such a list are cold-cache and serialised: compare shares, not absolute times.

DRAM traffic (``--metrics dram__bytes_read.sum,dram__bytes_write.sum --csv``)::

    python -m paper_2607_14530_gb300.ncu_summary traffic.csv --traffic OUT.json --workload W
        --scale S --map NAME=KERNEL [--map ...]

writes, for every trace name NAME mapped to a kernel, the mean DRAM bytes (read + write) per
launch of that kernel times S (the ratio of the benchmark's token count to the captured one:
every kernel's traffic is linear in the tokens), tagged with the hash of the kernel sources, so
that ``bench.py`` reports it only while the sources are unchanged.  With ``--forward TOKENS``
(the capture holding exactly one fwd+bwd step of TOKENS tokens, from its first launch) it also
stores, under ``_forward``, the measured forward DRAM bytes per token of one group: the launches
before the step's first ``k_restore`` (the backward's first kernel), divided by TOKENS.
"""
from __future__ import annotations

import csv
import hashlib
import glob
import io
import json
import os
import re
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _rows(path):
    with open(path) as f:
        text = f.read()
    start = text.find('"ID"')
    return list(csv.DictReader(io.StringIO(text[start:])))


def kernel_base(name: str) -> str:
    """`void xhc::<unnamed>::k_dx_tc<1>(CUtensorMap_st, ...)` -> `k_dx_tc<1>`."""
    name = name.replace("(anonymous namespace)", "").replace("<unnamed>", "")
    name = re.sub(r"\(.*$", "", name).replace("void ", "").strip()
    return name.split("::")[-1]


def load(path):
    out = []
    for r in _rows(path):
        if r.get("Metric Name") != "gpu__time_duration.sum":
            continue
        v = float(r["Metric Value"].replace(",", ""))
        unit = r.get("Metric Unit", "ns")
        scale = {"ns": 1e-6, "us": 1e-3, "usecond": 1e-3, "ms": 1.0, "msecond": 1.0, "nsecond": 1e-6}.get(unit, 1e-6)
        out.append((kernel_base(r["Kernel Name"]), v * scale))
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


def dram_bytes(path):
    """Mean DRAM bytes (read + write) per launch, per kernel."""
    unit_scale = {"byte": 1.0, "Kbyte": 1e3, "Mbyte": 1e6, "Gbyte": 1e9, "Tbyte": 1e12}
    per_launch = {}
    for r in _rows(path):
        m = r.get("Metric Name")
        if m not in ("dram__bytes_read.sum", "dram__bytes_write.sum"):
            continue
        v = float(r["Metric Value"].replace(",", "")) * unit_scale.get(r.get("Metric Unit", "byte"), 1.0)
        key = (r["ID"], kernel_base(r["Kernel Name"]))
        per_launch[key] = per_launch.get(key, 0.0) + v
    per = {}
    for (_, name), v in per_launch.items():
        per.setdefault(name, []).append(v)
    return {n: sum(v) / len(v) for n, v in per.items()}


def dram_launches(path):
    """[(launch id, kernel, DRAM bytes read + written)] in launch order."""
    unit_scale = {"byte": 1.0, "Kbyte": 1e3, "Mbyte": 1e6, "Gbyte": 1e9, "Tbyte": 1e12}
    per = {}
    for r in _rows(path):
        if r.get("Metric Name") not in ("dram__bytes_read.sum", "dram__bytes_write.sum"):
            continue
        v = float(r["Metric Value"].replace(",", "")) * unit_scale.get(r.get("Metric Unit", "byte"), 1.0)
        key = (int(r["ID"]), kernel_base(r["Kernel Name"]))
        per[key] = per.get(key, 0.0) + v
    return [(i, n, v) for (i, n), v in sorted(per.items())]


def forward_bytes(path):
    """(DRAM bytes of the launches before the first k_restore, number of those launches)."""
    tot, n = 0.0, 0
    for _, name, v in dram_launches(path):
        if name == "k_restore":
            return tot, n
        tot += v
        n += 1
    raise ValueError("no k_restore launch in the capture: it must hold a whole fwd+bwd step")


def csrc_hash():
    h = hashlib.sha256()
    for f in sorted(glob.glob(os.path.join(ROOT, "paper_2607_14530_gb300", "csrc", "*"))):
        with open(f, "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def main(argv):
    path = argv[1]
    if "--traffic" in argv:
        out = argv[argv.index("--traffic") + 1]
        wl = argv[argv.index("--workload") + 1]
        scale = float(argv[argv.index("--scale") + 1])
        maps = [argv[i + 1].split("=", 1) for i, a in enumerate(argv) if a == "--map"]
        per = dram_bytes(path)
        d = {}
        if os.path.exists(out):
            with open(out) as f:
                d = json.load(f)
        ent = d.setdefault(wl, {})
        sha = csrc_hash()
        for name, kern in maps:
            if kern in per:
                ent[name] = {"kernel": kern, "dram_bytes_per_launch": per[kern] * scale,
                             "captured_bytes_per_launch": per[kern], "scale": scale, "csrc_sha": sha}
        if "--forward" in argv:
            toks = int(argv[argv.index("--forward") + 1])
            fb, nl = forward_bytes(path)
            ent["_forward"] = {"dram_bytes_per_token": fb / toks, "captured_tokens": toks,
                               "launches": nl, "csrc_sha": sha}
            print(f"forward: {fb / 1e9:.4f} GB over {nl} launches = {fb / toks:.0f} bytes per token")
        with open(out, "w") as f:
            json.dump(d, f, indent=1, sort_keys=True)
        for n, v in sorted(per.items()):
            print(f"{n:28s} {v / 1e9:10.4f} GB per launch (captured)")
        return
    launches = load(path)
    if "--last" in argv:
        launches = launches[-int(argv[argv.index("--last") + 1]):]
    print(summarise(launches))


if __name__ == "__main__":
    main(sys.argv)
