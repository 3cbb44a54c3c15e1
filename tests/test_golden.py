"""Fixtures under tests/golden/.

worked_examples.json holds small problems whose results follow by hand from
the definition of attention (closed forms in e, written out with their
derivation); tiny_decode.json holds the oracle's outputs for the tiny decode
batch, written by tests/golden/make_golden.py. The oracle is checked against
the hand results and must reproduce its stored outputs bit for bit; on a GPU
the CUDA path is checked against both."""
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
import workloads as W

HERE = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
D, PAGE = 64, 16


def _bf16_bits(x: float) -> int:
    b = int(np.array([x], np.float32).view(np.uint32)[0])
    assert b & 0xFFFF == 0, f"{x} is not exact in bf16"
    return b >> 16


def _examples():
    with open(os.path.join(HERE, "worked_examples.json")) as f:
        return json.load(f)["examples"]


def _host_problem(ex):
    hq, hkv = ex["num_q_heads"], ex["num_kv_heads"]
    sl = np.asarray(ex["seq_lens"], np.int32)
    qsl = np.concatenate([[0], np.cumsum(ex["q_lens"])]).astype(np.int32)
    T = int(qsl[-1])
    q = np.zeros((T, hq, D), np.uint16)
    k_new = np.zeros((T, hkv, D), np.uint16)
    v_new = np.zeros((T, hkv, D), np.uint16)
    kc = np.zeros((ex["num_pages"], hkv, PAGE, D), np.uint16)
    vc = np.zeros_like(kc)
    for arr, key in ((q, "q"), (k_new, "k_new"), (v_new, "v_new")):
        for t, h, d, v in ex[key]:
            arr[t, h, d] = _bf16_bits(v)
    for arr, key in ((kc, "k_cache"), (vc, "v_cache")):
        for pg, h, s, d, v in ex[key]:
            arr[pg, h, s, d] = _bf16_bits(v)
    bt = np.asarray(ex["block_table"], np.int32)
    return dict(q=q, k_new=k_new, v_new=v_new, k_cache=kc, v_cache=vc, block_table=bt, seq_lens=sl,
                query_start_loc=qsl, window=ex["window"], scale=ex["scale"])


def _expected(ex, T, hq):
    out = np.zeros((T, hq, D))
    for t, h, d, v in ex["expect_out"]:
        out[t, h, d] = v
    lse = np.full((T, hq), np.nan)
    for t, h, v in ex["expect_lse"]:
        lse[t, h] = v
    return out, lse


@pytest.mark.parametrize("ex", _examples(), ids=lambda e: e["name"])
def test_oracle_reproduces_hand_derived_results(ex):
    p = _host_problem(ex)
    kc, vc = oracle.kv_append(p["k_new"], p["v_new"], p["k_cache"], p["v_cache"], p["block_table"], p["seq_lens"],
                              p["query_start_loc"])
    out, lse = oracle.paged_attention(p["q"], kc, vc, p["block_table"], p["seq_lens"], p["query_start_loc"],
                                      p["window"], p["scale"])
    ref_out, ref_lse = _expected(ex, out.shape[0], out.shape[1])
    got = oracle.bf16_bits_to_float(out).astype(np.float64)
    # one rounding to bf16 (half an ulp) and nothing else
    assert np.all(np.abs(got - ref_out) <= np.abs(ref_out) * 2.0**-8), ex["name"]
    listed = ~np.isnan(ref_lse)
    assert np.all(np.abs(lse[listed] - ref_lse[listed]) <= 1e-6 * np.maximum(1.0, np.abs(ref_lse[listed])))


def test_oracle_reproduces_its_stored_tiny_decode_outputs():
    with open(os.path.join(HERE, "tiny_decode.json")) as f:
        g = json.load(f)
    b = W.config_tiny()
    h = W.host_inputs(b)
    kc, vc = oracle.kv_append(h["k_new"], h["v_new"], h["k_cache"], h["v_cache"], h["block_table"],
                              h["seq_lens"], h["query_start_loc"])
    out, lse = oracle.paged_attention(h["q"], kc, vc, h["block_table"], h["seq_lens"], h["query_start_loc"],
                                      h["sliding_window"], h["softmax_scale"])
    assert list(out.shape) == g["shape_out"]
    assert np.array_equal(out.reshape(-1), np.asarray(g["out_bf16_bits"], np.uint16))
    assert np.array_equal(lse.reshape(-1), np.asarray(g["lse"], np.float32))


# ------------------------------------------------------------------ GPU


def _run_cuda(p, hq, hkv):
    from paper_2608_22167_gb300 import mcpu

    dev = torch.device("cuda")

    def bf(a):
        return torch.from_numpy(a.astype(np.int16)).view(torch.bfloat16).to(dev)

    q, k_new, v_new = bf(p["q"]), bf(p["k_new"]), bf(p["v_new"])
    kc, vc = bf(p["k_cache"]), bf(p["v_cache"])
    bt = torch.from_numpy(p["block_table"]).to(dev)
    sl = torch.from_numpy(p["seq_lens"]).to(dev)
    qsl = torch.from_numpy(p["query_start_loc"]).to(dev)
    d = mcpu.dims(q, kc, bt, sl)
    ws = mcpu.new_workspace(d, dev)
    out = torch.full_like(q, float("nan"))
    lse = torch.full(q.shape[:2], float("nan"), dtype=torch.float32, device=dev)
    mcpu.mcpu_kv_append(k_new, v_new, kc, vc, bt, sl, qsl, mcpu.status_word(ws))
    mcpu.mcpu_paged_attention_forward(q, kc, vc, bt, sl, qsl, p["window"], p["scale"], out, lse, ws)
    code, bits = mcpu.mcpu_read_device_status(ws)
    assert code == 0, bits
    return out.float().cpu().numpy(), lse.cpu().numpy()


@pytest.mark.gpu
@pytest.mark.parametrize("ex", _examples(), ids=lambda e: e["name"])
def test_cuda_path_reproduces_hand_derived_results(ex):
    p = _host_problem(ex)
    out, lse = _run_cuda(p, ex["num_q_heads"], ex["num_kv_heads"])
    ref_out, ref_lse = _expected(ex, out.shape[0], out.shape[1])
    # P is rounded to bf16 before P.V (half an ulp, 2^-9) and out once more
    assert np.all(np.abs(out - ref_out) <= np.abs(ref_out) * 2.0**-7 + 1e-6), ex["name"]
    listed = ~np.isnan(ref_lse)
    assert np.all(np.abs(lse[listed] - ref_lse[listed]) <= 1e-3)


@pytest.mark.gpu
def test_cuda_path_matches_stored_tiny_decode_outputs():
    from _gpu import LSE_ABS, OUT_ABS, OUT_REL

    with open(os.path.join(HERE, "tiny_decode.json")) as f:
        g = json.load(f)
    b = W.config_tiny()
    h = W.host_inputs(b)
    p = dict(q=h["q"], k_new=h["k_new"], v_new=h["v_new"], k_cache=h["k_cache"], v_cache=h["v_cache"],
             block_table=h["block_table"], seq_lens=h["seq_lens"], query_start_loc=h["query_start_loc"],
             window=h["sliding_window"], scale=h["softmax_scale"])
    out, lse = _run_cuda(p, b.num_q_heads, b.num_kv_heads)
    ref = oracle.bf16_bits_to_float(np.asarray(g["out_bf16_bits"], np.uint16)).reshape(g["shape_out"])
    err = np.abs(out - ref)
    assert err.max() <= OUT_ABS and err.max() / np.abs(ref).max() <= OUT_REL
    assert np.abs(lse.reshape(-1) - np.asarray(g["lse"], np.float32)).max() <= LSE_ABS
