"""Summarise parity logs (the KINT_PARITY_LOG files that tests/parity.check appends to) as a
markdown table with one row per case, plus a compact JSON record per case.

    python tests/parity_report.py LOG.jsonl [LOG2.jsonl ...] > summary.md
"""
from __future__ import annotations

import json
import sys

CALIB = {0: "MinMax", 1: "FWM", 2: "softmax", 3: "FWM-resolved", 4: "exp-FP8", 5: "exp-BF16"}
RECON = {0: "LERP", 1: "Nearest"}
STE = {0: "Weight", 1: "Prob"}
GRAD = {0: "full", 1: "detach", 2: "max_only", 3: "min_only", 4: "detach_proj"}


def _fmt(x):
    return "—" if x is None else f"{x:.2g}"


def main(paths):
    recs = []
    for path in paths:
        with open(path) as fh:
            recs += [json.loads(line) for line in fh if line.strip()]
    print("| case | prec | B,H,T,d | operator | flip fraction | arg-max flips | O | dQ | dK | dV | worst (tol) | "
          "zero-sum GPU median / max | oracle median |")
    print("|---|---|---|---|---|---|---|---|---|---|---|---|---|")
    compact = []
    for r in recs:
        c = r["cfg"]
        op = f"{CALIB[c['calib']]} K={c['Kint']} {RECON[c['recon']]} {STE[c['ste']]}-STE {GRAD[c['grad']]}"
        e = r["errors"]
        worst = max(e.items(), key=lambda kv: kv[1]) if e else ("—", None)
        zg, zo = r.get("zero_sum_gpu", {}), r.get("zero_sum_oracle", {})
        name = r["case"].split("::")[-1]
        print(f"| {name} | {r['prec']} | {','.join(map(str, r['shape']))} | {op} | {_fmt(r['flip_fraction'])} | "
              f"{r['arg_max_flips']} | {_fmt(e.get('O'))} | {_fmt(e.get('dQ'))} | {_fmt(e.get('dK'))} | "
              f"{_fmt(e.get('dV'))} | {worst[0]} {_fmt(worst[1])} ({r['tol']:g}) | {_fmt(zg.get('median'))} / "
              f"{_fmt(zg.get('max'))} | {_fmt(zo.get('median'))} |")
        compact.append({"case": name, "prec": r["prec"], "flip": float(f"{r['flip_fraction']:.3g}"),
                        "amax_flips": r["arg_max_flips"],
                        "err": {k: float(f"{e[k]:.3g}") for k in ("O", "dQ", "dK", "dV") if k in e},
                        "zs_gpu_median": None if zg.get("median") is None else float(f"{zg['median']:.3g}")})
    print()
    print("Compact records (one JSON object per case):")
    print()
    print("```")
    for c in compact:
        print(json.dumps(c, separators=(",", ":")))
    print("```")


if __name__ == "__main__":
    main(sys.argv[1:])
