"""Writes tests/golden/config_summaries.json: for each of the five workloads,
the SHA-256 of the generated trace bytes and summary statistics computed by
the CPU oracle only (never by the CUDA path).

The parity tests re-generate and re-run the oracle on whatever host they run
on and compare with this file, which catches generator or oracle drift
between machines (x86-64 here, AArch64 on the GPU hosts).

    python tests/golden/make_config_summaries.py
"""
import json
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

import numpy as np  # noqa: E402

import oracle  # noqa: E402
import tracegen  # noqa: E402


def summarize(k: int) -> dict:
    ts = tracegen.config(k)
    prof, lb, st_p = oracle.live_profile(ts)
    out = {
        "name": ts.name,
        "sha256": tracegen.digest(ts),
        "n_traces": ts.n_traces,
        "n_tensors": ts.n_tensors,
        "pairs": ts.pairs(),
        "profile_sum": int(prof.sum()),
        "peak_lb_sum": int(lb.sum()),
        "status_ok": bool((st_p == 0).all()),
    }
    for pol, key in ((oracle.FIT_FIRST, "first"), (oracle.FIT_BEST, "best")):
        off, pk, st = oracle.plan_greedy_by_size(ts, pol)
        v, _, st_v = oracle.validate_plan(ts, off)
        out[f"{key}_offsets_sum"] = int(off.sum())
        out[f"{key}_plan_peak_sum"] = int(pk.sum())
        out[f"{key}_all_valid"] = bool((v == 1).all())
        out["status_ok"] = out["status_ok"] and bool((st == 0).all() and (st_v == 0).all())
    return out


def main():
    res = {"about": "Written by tests/golden/make_config_summaries.py from tracegen + oracle only.",
           "configs": [summarize(k) for k in range(5)]}
    with open(os.path.join(HERE, "config_summaries.json"), "w") as f:
        json.dump(res, f, indent=2)
        f.write("\n")


if __name__ == "__main__":
    main()
