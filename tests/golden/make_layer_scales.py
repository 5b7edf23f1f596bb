"""Write tests/golden/layer_scales.json: the frozen int8 output scales of
one encoder layer's chain (QKV, attention context, attention output, FFN1,
FFN2) on the seeded layer inputs (synth.encoder_layer: M = 8 x 384 tokens,
80% block sparsity).

Each scale is max |y| / 127 of the stage's unquantised output, computed by
the CPU oracle only (oracle.calibrate_chain): post-training calibration of
a static per-tensor scale, as the paper's quantisation step does with its
calibration set (Sec. 2).  Both the oracle chain and the GPU chain then use
these constants.  Run: python tests/golden/make_layer_scales.py
"""
import json
import os
import sys
import time

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
import synth  # noqa: E402

BATCH, SEQ = 8, 384


def main():
    t0 = time.time()
    weights, x0 = synth.encoder_layer()
    assert x0.shape[0] == BATCH * SEQ
    scales = oracle.calibrate_chain(x0, weights, BATCH, SEQ, threads=os.cpu_count() or 8)
    doc = {"source": "oracle.calibrate_chain on synth.encoder_layer() (seeded), scale = max|y| / 127 in fp32",
           "batch": BATCH, "seq": SEQ, "sparsity": 0.80, "scales": scales}
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "layer_scales.json")
    with open(path, "w") as f:
        json.dump(doc, f, indent=1)
        f.write("\n")
    print(json.dumps(scales), f"{time.time() - t0:.1f} s")


if __name__ == "__main__":
    main()
