"""Write the oracle's results for the full-size workloads to tests/golden/oracle_energies.json.

Calls only ``oracle/`` (the fp64 CPU restatement of the method) and the seeded generators; nothing here comes
from the CUDA path. The GPU tests compare the library's final energy with these values (|dE| <= 1e-4) at sizes
where rerunning the oracle inside a test would take minutes.

    python tests/golden/make_golden.py [workload names...]      # default: all, plus decoder layers 0, 17, 35

Decoder matrices are named L<layer>.<projection> (e.g. L17.gate); any of the 36 layers can be asked for.
"""
import json
import os
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

from oracle import externd_oracle as O          # noqa: E402
from paper_2607_13511_gb300 import workloads as W  # noqa: E402

OUT = os.path.join(os.path.dirname(os.path.abspath(__file__)), "oracle_energies.json")


def run(wl: W.Workload) -> dict:
    A = wl.matrix()
    h = wl.weights()
    t0 = time.time()
    res = O.decompose(A, wl.mu, wl.tau, wl.block, wl.iters, h)
    seconds = time.time() - t0
    return {
        "m": wl.m, "n": wl.n, "mu": wl.mu, "tau": wl.tau, "block": wl.block, "iters": wl.iters,
        "weighted": wl.weighted, "k": int(res.D.size),
        "energy": res.energy,
        "energy_reconstructed": O.energy(A, res.B, res.D, res.C, h),
        "trace": [float(x) for x in res.trace],
        "zero_fraction_B": float((res.B == 0).mean()),
        "zero_fraction_C": float((res.C == 0).mean()),
        "oracle_seconds": seconds,
    }


def main(names):
    table = json.load(open(OUT)) if os.path.exists(OUT) else {}
    todo = {w.name: w for w in W.WORKLOADS.values()}
    decoder = {w.name: w for w in W.decoder_conversion()}
    todo.update({name: wl for name, wl in decoder.items() if name.split(".")[0] in ("L0", "L17", "L35")})
    for name in names or list(todo):
        todo.setdefault(name, decoder.get(name))
        print(f"{name} ...", flush=True)
        table[name] = run(todo[name])
        print(f"  E = {table[name]['energy']:.8f} in {table[name]['oracle_seconds']:.1f} s", flush=True)
        with open(OUT, "w") as f:
            json.dump({"source": "oracle/externd_oracle.py via tests/golden/make_golden.py", **table}, f, indent=1)
            f.write("\n")


if __name__ == "__main__":
    main([a for a in sys.argv[1:]])
