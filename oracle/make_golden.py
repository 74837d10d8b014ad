"""Writes tests/golden/*.json: oracle results at the benchmark workloads' full sizes.

TEST INFRASTRUCTURE.  Calls only the CPU oracle (oracle/) on inputs drawn by the
seeded generator; nothing here touches the CUDA path.  Run once, commit the JSON:

    python oracle/make_golden.py large        # N=6, 24^6 candidates, full enumeration
    python oracle/make_golden.py stress       # N=8, two index ranges of 2^24 of 16^8
"""
from __future__ import annotations

import json
import os
import sys
import time

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

from oracle.oracle import Oracle, build  # noqa: E402
from paper_2609_02109_gb300 import workload as W  # noqa: E402

GOLDEN = os.path.join(ROOT, "tests", "golden")


def _run(name, prob, ranges, k):
    o = Oracle(prob)
    out = {"workload": name, "generator": "paper_2609_02109_gb300.workload", "k": k, "ranges": []}
    for lo, hi in ranges:
        t = time.time()
        ti, ts, cnt = o.exhaustive(k, lo=lo, hi=hi)
        out["ranges"].append({"lo": lo, "hi": hi, "count": cnt, "topk_idx": [int(i) for i in ti],
                              "topk_score": [float(s) for s in ts], "seconds": round(time.time() - t, 1)})
        print(name, lo, hi, cnt, ti[:3], ts[:3], f"{time.time() - t:.1f}s", flush=True)
    return out


def main(which):
    build()
    os.makedirs(GOLDEN, exist_ok=True)
    if which == "large":
        prob = W.large(precision="fp32")
        res = _run("large: N=6 x 24 options, 12->64->64->2, seed 3", prob, [(0, 24 ** 6)], 64)
    elif which == "stress":
        prob = W.stress(precision="fp32")
        n = 16 ** 8
        res = _run("stress: N=8 x 16 options, 20->128->128->2, soft latency, seed 4", prob,
                   [(0, 1 << 24), (n - (1 << 24), n)], 64)
    else:
        raise SystemExit("usage: make_golden.py large|stress")
    with open(os.path.join(GOLDEN, f"{which}.json"), "w") as f:
        json.dump(res, f, indent=1)


if __name__ == "__main__":
    main(sys.argv[1])
