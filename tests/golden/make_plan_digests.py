"""Write tests/golden/plan_digests.txt: the oracle's whole plan (Algorithm 1 with
the workload's starts and rounds, default orders, safeguards where they apply)
on the paper-scale and stress workloads, too large for the oracle to run inside
the test suite.  Each line holds the workload, the objective, the returned
candidate index and the SHA-256 of the placement bytes ([W][n] uint8, 1 =
resident).  Calls only oracle/ and the seeded workload generator.

usage: python tests/golden/make_plan_digests.py [cfg ...] [--threads N]
"""
import argparse
import hashlib
import os
import sys
import time

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

import oracle  # noqa: E402
from paper_2608_01655_gb300 import workloads as wl  # noqa: E402

OUT = os.path.join(HERE, "plan_digests.txt")


def digest(placement) -> str:
    return hashlib.sha256(placement.astype("uint8").tobytes()).hexdigest()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("cfgs", nargs="*", type=int, default=[3, 4])
    ap.add_argument("--threads", type=int, default=os.cpu_count())
    args = ap.parse_args()
    lines = {}
    if os.path.exists(OUT):
        for line in open(OUT):
            if line.strip() and not line.startswith("#"):
                lines[line.split()[0]] = line.rstrip("\n")
    for cfg in args.cfgs:
        inst = wl.make(cfg)
        prob = oracle.Problem.from_instance(inst)
        t0 = time.time()
        r = oracle.plan(prob, inst.starts, inst.rounds, threads=args.threads)
        lines[inst.name] = f"{inst.name} {r.objective} {r.best_start} {digest(r.placement)}"
        print(f"{inst.name}: objective {r.objective} best {r.best_start} in {time.time() - t0:.0f} s", flush=True)
        with open(OUT, "w") as f:
            f.write("# Oracle plans (Algorithm 1, default orders, the workload's starts and rounds)\n")
            f.write("# written by tests/golden/make_plan_digests.py; columns: workload objective\n")
            f.write("# returned-candidate sha256(placement [W][n] uint8)\n")
            for name in sorted(lines):
                f.write(lines[name] + "\n")


if __name__ == "__main__":
    main()
