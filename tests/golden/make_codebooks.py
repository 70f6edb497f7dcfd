"""Write tests/golden/codebooks.json from the oracle alone.

Stores the oracle's Lloyd-Max codebooks (Sec. II-B step 3) for the d = 1536
workloads at b in {2, 3, 4, 8} for both marginals, so tests do not rerun the
slow 8-bit iteration.  Calls nothing but oracle/.

    python tests/golden/make_codebooks.py
"""
import json
import os
import sys
import time

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

import oracle  # noqa: E402


def main() -> None:
    out = {"source": "oracle.codebook (plain Lloyd-Max, float64)", "entries": []}
    for marginal in ("beta", "gauss"):
        for bits in (2, 3, 4, 8):
            t0 = time.time()
            cb = oracle.codebook(1536, bits, marginal)
            out["entries"].append({
                "d": 1536, "bits": bits, "marginal": marginal,
                "centroids": [float(v) for v in cb.centroids],
                "boundaries": [float(v) for v in cb.boundaries],
                "distortion": cb.distortion, "iterations": cb.iterations,
            })
            print(marginal, bits, cb.iterations, f"{time.time() - t0:.1f}s", flush=True)
    with open(os.path.join(HERE, "codebooks.json"), "w") as f:
        json.dump(out, f, indent=1)


if __name__ == "__main__":
    main()
