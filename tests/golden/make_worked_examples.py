"""Writes worked_examples.json: small attention problems whose results follow
by hand from the definition (softmax attention with causal and window masks,
q head h reading kv head h // g). Inputs are sparse and exact in bf16; every
expected value is a closed form in e, evaluated here with the math module
only (no oracle, no GPU). Run from the repository root:
    python tests/golden/make_worked_examples.py
"""
import json
import math
import os

HERE = os.path.dirname(os.path.abspath(__file__))
e = math.e


def one_hot(dim):
    return dim


examples = []

# A. three keys, full context: q = 8 e0, k_j = j e0, v_j = e_j, scale 1/8 ->
# scores (0, 1, 2); out dims 0..2 = (1, e, e^2) / (1 + e + e^2).
zA = 1 + e + e * e
examples.append(dict(
    name="three_keys_full_context",
    derivation="scores s_j = (1/8)(8 e0).(j e0) = j for j = 0, 1, 2; out = sum_j e^{s_j} v_j / Z, Z = 1 + e + e^2; "
               "lse = ln Z",
    num_q_heads=1, num_kv_heads=1, seq_lens=[3], q_lens=[1], window=0, scale=0.125,
    num_pages=1, block_table=[[0]],
    q=[[0, 0, 0, 8.0]],
    k_cache=[[0, 0, 1, 0, 1.0], [0, 0, 2, 0, 2.0]],
    v_cache=[[0, 0, 0, 0, 1.0], [0, 0, 1, 1, 1.0]],
    k_new=[[0, 0, 0, 2.0]], v_new=[[0, 0, 2, 1.0]],
    expect_out=[[0, 0, 0, 1 / zA], [0, 0, 1, e / zA], [0, 0, 2, e * e / zA]],
    expect_lse=[[0, 0, math.log(zA)]],
))

# B. the same with a window of 2 keys: key 0 is out of the window.
zB = e + e * e
examples.append(dict(
    name="three_keys_window_2",
    derivation="window W = 2 keeps keys j with 2 - j < 2, i.e. j = 1, 2; Z = e + e^2; out dims 1, 2 = "
               "(e, e^2) / Z = (1, e) / (1 + e); lse = ln Z = 1 + ln(1 + e)",
    num_q_heads=1, num_kv_heads=1, seq_lens=[3], q_lens=[1], window=2, scale=0.125,
    num_pages=1, block_table=[[0]],
    q=[[0, 0, 0, 8.0]],
    k_cache=[[0, 0, 1, 0, 1.0], [0, 0, 2, 0, 2.0]],
    v_cache=[[0, 0, 0, 0, 1.0], [0, 0, 1, 1, 1.0]],
    k_new=[[0, 0, 0, 2.0]], v_new=[[0, 0, 2, 1.0]],
    expect_out=[[0, 0, 1, e / zB], [0, 0, 2, e * e / zB]],
    expect_lse=[[0, 0, math.log(zB)]],
))

# C. an appended chunk of two tokens (positions 1, 2), causal inside it.
z1 = 1 + e
examples.append(dict(
    name="append_chunk_of_two_causal",
    derivation="S = 3, L = 2: token 0 sits at position 1 and sees keys 0, 1 (scores 0, 1): out dims 0, 1 = "
               "(1, e) / (1 + e), lse = ln(1 + e); token 1 at position 2 sees keys 0..2 as in example A. The "
               "chunk's keys and values enter the cache through the KV append (k_new, v_new)",
    num_q_heads=1, num_kv_heads=1, seq_lens=[3], q_lens=[2], window=0, scale=0.125,
    num_pages=1, block_table=[[0]],
    q=[[0, 0, 0, 8.0], [1, 0, 0, 8.0]],
    k_cache=[], v_cache=[[0, 0, 0, 0, 1.0]],
    k_new=[[0, 0, 0, 1.0], [1, 0, 0, 2.0]], v_new=[[0, 0, 1, 1.0], [1, 0, 2, 1.0]],
    expect_out=[[0, 0, 0, 1 / z1], [0, 0, 1, e / z1],
                [1, 0, 0, 1 / zA], [1, 0, 1, e / zA], [1, 0, 2, e * e / zA]],
    expect_lse=[[0, 0, math.log(z1)], [1, 0, math.log(zA)]],
))

# D. grouped query heads: two q heads read one kv head with opposite queries.
examples.append(dict(
    name="gqa_two_heads_one_kv_head",
    derivation="g = 2: q heads 0 and 1 read kv head 0. Keys k0 = 0, k1 = e0; q0 = 8 e0 gives scores (0, 1), "
               "q1 = -8 e0 gives (0, -1). Head 0: out dims 0, 1 = (1, e) / (1 + e), lse = ln(1 + e); head 1: "
               "(1, 1/e) / (1 + 1/e) = (e, 1) / (1 + e), lse = ln(1 + 1/e)",
    num_q_heads=2, num_kv_heads=1, seq_lens=[2], q_lens=[1], window=0, scale=0.125,
    num_pages=1, block_table=[[0]],
    q=[[0, 0, 0, 8.0], [0, 1, 0, -8.0]],
    k_cache=[], v_cache=[[0, 0, 0, 0, 1.0]],
    k_new=[[0, 0, 0, 1.0]], v_new=[[0, 0, 1, 1.0]],
    expect_out=[[0, 0, 0, 1 / z1], [0, 0, 1, e / z1], [0, 1, 0, e / z1], [0, 1, 1, 1 / z1]],
    expect_lse=[[0, 0, math.log(z1)], [0, 1, math.log(1 + 1 / e)]],
))

# E. seventeen keys over two physical pages listed in reverse order; all
# scores equal, so out is the plain mean of v: v_j = (j + 1) e0 -> 9.
examples.append(dict(
    name="seventeen_equal_scores_two_pages",
    derivation="all keys are 0, so every score is 0 and the weights are 1/17: out dim 0 = (1 + ... + 17) / 17 = 9, "
               "lse = ln 17. Logical page 0 is physical page 1 and logical page 1 is physical page 0",
    num_q_heads=1, num_kv_heads=1, seq_lens=[17], q_lens=[1], window=0, scale=0.125,
    num_pages=2, block_table=[[1, 0]],
    q=[[0, 0, 0, 8.0]],
    k_cache=[],
    v_cache=[[1, 0, j, 0, float(j + 1)] for j in range(16)],
    k_new=[], v_new=[[0, 0, 0, 17.0]],
    expect_out=[[0, 0, 0, 9.0]],
    expect_lse=[[0, 0, math.log(17)]],
))

if __name__ == "__main__":
    doc = {
        "about": "hand-derived attention results; sparse inputs: q, k_new, v_new entries are [token, head, dim, "
                 "value], k_cache, v_cache entries [page, kv head, slot, dim, value]; all other inputs are 0. "
                 "expect_out lists [token, q head, dim, value] and every unlisted output is 0; expect_lse lists "
                 "[token, q head, natural-log value]. head_dim 64, page size 16",
        "examples": examples,
    }
    path = os.path.join(HERE, "worked_examples.json")
    with open(path, "w") as f:
        json.dump(doc, f, indent=1)
        f.write("\n")
    print(path)
