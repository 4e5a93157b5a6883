"""Write tests/golden/tiny_seed0.json: the oracle's output on the tiny
workload (seed 0). Calls only the oracle and the input generator; rerun it
only when a change to the oracle's arithmetic is justified by the paper."""
import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
import synth  # noqa: E402


def main():
    w = synth.tiny(0)
    f, c, n = oracle.voxelize_roi(w.points, w.sweep_offsets, w.sweep_tf, w.rois, w.roi_margin,
                                  w.voxel_size, w.pc_range, w.max_pts_per_voxel, w.max_voxels)
    doc = {
        "what": "oracle output, tiny workload seed 0 (20,000 uniform points, 4 ROIs, "
                "512x512x1 pillars, K=10, max 16,000 voxels); Alg. 1 with Eq. 1 boxes",
        "coords": c.tolist(),
        "counts": n.tolist(),
        "feats_hex": [[float.hex(float(v)) for v in row] for row in f],
    }
    with open(os.path.join(os.path.dirname(os.path.abspath(__file__)), "tiny_seed0.json"), "w") as fh:
        json.dump(doc, fh, separators=(",", ":"))


if __name__ == "__main__":
    main()
