"""Writes the oracle-derived fixtures of this folder.

Only the CPU oracle (oracle/) and the seeded input generator (workloads.py)
are used here; nothing comes from the CUDA path. Run from the repository
root:  python tests/golden/make_golden.py
"""
import json
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
import workloads as W  # noqa: E402


def tiny_decode():
    """Every output of the tiny decode batch (4 rows with KV lengths
    {17, 64, 129, 300}, 8 q / 2 kv heads, seed 1001): out as bf16 bit
    patterns, lse as float32."""
    b = W.config_tiny()
    h = W.host_inputs(b)
    kc, vc = oracle.kv_append(h["k_new"], h["v_new"], h["k_cache"], h["v_cache"], h["block_table"],
                              h["seq_lens"], h["query_start_loc"])
    out, lse = oracle.paged_attention(h["q"], kc, vc, h["block_table"], h["seq_lens"], h["query_start_loc"],
                                      h["sliding_window"], h["softmax_scale"])
    return {
        "what": "oracle outputs of the tiny decode batch (workloads.config_tiny, seed 1001), KV append applied",
        "shape_out": list(out.shape),
        "out_bf16_bits": [int(x) for x in out.reshape(-1)],
        "lse": [float(x) for x in lse.reshape(-1)],
    }


if __name__ == "__main__":
    path = os.path.join(HERE, "tiny_decode.json")
    with open(path, "w") as f:
        json.dump(tiny_decode(), f, separators=(",", ":"))
        f.write("\n")
    print(path)
