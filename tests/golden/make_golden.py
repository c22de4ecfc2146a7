"""Writes tests/golden/oracle_tiny.json: a tiny RMAT graph, two minibatches
of targets, and the oracle's outputs and blocks-touched statistics for them.

Calls only the oracle (and the seeded input generator for the graph, which is
stored in the fixture itself).  Re-run only when a change to the oracle's
arithmetic is justified by the paper; the fixture freezes conventions the
paper leaves open (Philox key layout, bit order of the 64-bit draw).
"""
import json
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

import oracle  # noqa: E402
from agnes_inputs import synth  # noqa: E402

N, DEG, SEED = 256, 6, 11
FANOUTS = [3, 2]
ADJ_BB, FEAT_BB = 64, 64
RNG_SEED, FIRST_GID = 0xC0FFEE, 40


def main():
    import torch
    off, ind = synth.rmat_csr(N, DEG, 0.57, 0.19, 0.19, SEED, offsets_dtype=torch.int32)
    feats = (np.arange(N * 4, dtype=np.int64).reshape(N, 4) % 997).astype(np.float32)
    targets = synth.permutation(N, 5)[:16].view(2, 8).numpy().astype(np.int32)
    g = oracle.Graph(off.numpy(), ind.numpy(), feats)
    mbs, stats = oracle.hyperbatch(g, targets, FANOUTS, RNG_SEED, FIRST_GID, True, ADJ_BB, FEAT_BB)
    out = {
        "note": "oracle outputs for a tiny RMAT graph; written by make_golden.py",
        "offsets": off.tolist(), "indices": ind.tolist(), "features": feats.tolist(),
        "targets": targets.tolist(), "fanouts": FANOUTS, "seed": RNG_SEED,
        "first_gid": FIRST_GID, "adj_block_bytes": ADJ_BB, "feat_block_bytes": FEAT_BB,
        "stats": stats,
        "minibatches": [{
            "nodes": mb["nodes"].tolist(),
            "hops": [{"num_dst": h["num_dst"], "indptr": h["indptr"].tolist(),
                      "col": h["col"].tolist()} for h in mb["hops"]],
        } for mb in mbs],
    }
    with open(os.path.join(HERE, "oracle_tiny.json"), "w") as f:
        json.dump(out, f, separators=(",", ":"))
        f.write("\n")


if __name__ == "__main__":
    main()
