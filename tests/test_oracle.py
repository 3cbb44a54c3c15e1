"""Pins of the CPU oracle against facts that do not come from the oracle.

Each test checks ``oracle/`` against something independent of it: a second
brute-force formulation (numpy fp64, dense mask), a library routine
(torch's scaled_dot_product_attention in fp64), closed forms (one visible
key, q = 0, constant values), invariances of the definition (physical page
relabelling, paging itself, head grouping, causal and window locality) and
the log-sum-exp identity that split-KV merging relies on. A dropped term, a
wrong sign or index or a transposed operand in the oracle fails at least one.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from oracle import brute
import workloads as W


def _run_oracle(h, window=None):
    return oracle.paged_attention(
        h["q"], h["k_cache"], h["v_cache"], h["block_table"], h["seq_lens"], h["query_start_loc"],
        h["sliding_window"] if window is None else window, h["softmax_scale"],
    )


def _f(bits):
    return oracle.bf16_bits_to_float(bits).astype(np.float64)


def _assert_close_to_exact(out_bits, lse, ref_out, ref_lse):
    """Oracle vs an unrounded fp64 reference: out may differ by its one final
    rounding to bf16 (half an ulp, 2^-9 relative); lse by float32 rounding."""
    o = _f(out_bits)
    bound = np.abs(ref_out) * 2.0**-8 + 1e-30
    assert np.all(np.abs(o - ref_out) <= bound), np.max(np.abs(o - ref_out) - bound)
    fin = np.isfinite(ref_lse)
    assert np.array_equal(fin, np.isfinite(lse))
    assert np.all(np.abs(lse[fin] - ref_lse[fin]) <= 1e-6 * np.maximum(1.0, np.abs(ref_lse[fin])))


# ---------------------------------------------------------------- rounding


def test_bf16_rounding_matches_torch_rne():
    rng = np.random.default_rng(0)
    xs = np.concatenate([
        rng.standard_normal(2000).astype(np.float32),
        (rng.standard_normal(500) * 1e-38).astype(np.float32),  # subnormal range
        (rng.standard_normal(500) * 1e30).astype(np.float32),
    ])
    ref = torch.from_numpy(xs).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = np.array([oracle.double_to_bf16(float(x)) for x in xs], np.uint16)
    assert np.array_equal(got, ref)


def test_bf16_rounding_ties_to_even():
    # 1 + 2^-8 is halfway between 1 and 1 + 2^-7: even mantissa wins (1.0).
    assert oracle.double_to_bf16(1.0 + 2.0**-8) == 0x3F80
    # 1 + 3 * 2^-8 is halfway between 1 + 2^-7 (odd) and 1 + 2^-6 (even).
    assert oracle.double_to_bf16(1.0 + 3 * 2.0**-8) == 0x3F82
    # Just above a tie rounds up.
    assert oracle.double_to_bf16(1.0 + 2.0**-8 + 2.0**-30) == 0x3F81
    assert oracle.double_to_bf16(-2.0) == 0xC000
    assert oracle.double_to_bf16(0.0) == 0x0000
    assert oracle.double_to_bf16(2.0**200) == 0x7F80  # overflow -> +inf


# ---------------------------------------------------------- brute force


def test_tiny_config_matches_brute_force():
    b = W.config_tiny()
    h = W.host_inputs(b)
    out, lse = _run_oracle(h)
    ref_out, ref_lse = brute.attention(
        h["q"], h["k_cache"], h["v_cache"], h["block_table"], h["seq_lens"], h["query_start_loc"],
        h["sliding_window"], h["softmax_scale"],
    )
    _assert_close_to_exact(out, lse, ref_out, ref_lse)


@pytest.mark.parametrize("seed", range(40))
def test_fuzz_matches_brute_force(seed):
    b = W.fuzz_batch(seed)
    h = W.host_inputs(b)
    kc, vc = oracle.kv_append(h["k_new"], h["v_new"], h["k_cache"], h["v_cache"], h["block_table"],
                              h["seq_lens"], h["query_start_loc"])
    h["k_cache"], h["v_cache"] = kc, vc
    out, lse = _run_oracle(h)
    ref_out, ref_lse = brute.attention(h["q"], kc, vc, h["block_table"], h["seq_lens"],
                                       h["query_start_loc"], h["sliding_window"], h["softmax_scale"])
    _assert_close_to_exact(out, lse, ref_out, ref_lse)


@pytest.mark.parametrize("seed", range(8))
def test_peaked_fuzz_matches_brute_force(seed):
    rng = np.random.default_rng(100 + seed)
    B = int(rng.integers(1, 6))
    S = rng.integers(2, 200, size=B)
    L = np.minimum(S, rng.integers(1, 40, size=B))
    b = W.build_batch("peaked", 500 + seed, S, L, 16, 2, layer_windows=(int(rng.choice([0, 32])),), peaked=True)
    h = W.host_inputs(b)
    out, lse = _run_oracle(h)
    ref_out, ref_lse = brute.attention(h["q"], h["k_cache"], h["v_cache"], h["block_table"], h["seq_lens"],
                                       h["query_start_loc"], h["sliding_window"], h["softmax_scale"])
    _assert_close_to_exact(out, lse, ref_out, ref_lse)


# ------------------------------------------------------- library routine


@pytest.mark.parametrize("seed", [3, 11, 29])
def test_matches_torch_sdpa_fp64(seed):
    b = W.fuzz_batch(seed)
    h = W.host_inputs(b)
    out, lse = _run_oracle(h)
    qf = torch.from_numpy(brute.bits_to_f64(h["q"]))
    g = b.num_q_heads // b.num_kv_heads
    for r in range(b.num_seqs):
        S = int(h["seq_lens"][r])
        t0, t1 = int(h["query_start_loc"][r]), int(h["query_start_loc"][r + 1])
        if t1 == t0:
            continue
        k, v = brute.dense_kv(h["k_cache"], h["v_cache"], h["block_table"][r], S, 16)
        kt = torch.from_numpy(k).permute(1, 0, 2).repeat_interleave(g, 0)  # [Hq, S, D]
        vt = torch.from_numpy(v).permute(1, 0, 2).repeat_interleave(g, 0)
        qt = qf[t0:t1].permute(1, 0, 2)  # [Hq, L, D]
        p = torch.arange(S - (t1 - t0), S)[:, None]
        j = torch.arange(S)[None, :]
        mask = j <= p
        if h["sliding_window"] > 0:
            mask &= (p - j) < h["sliding_window"]
        ref = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, attn_mask=mask, scale=h["softmax_scale"])
        ref_out = ref.permute(1, 0, 2).numpy()
        o = _f(out[t0:t1])
        assert np.all(np.abs(o - ref_out) <= np.abs(ref_out) * 2.0**-8 + 1e-12)
        # lse from the library's own logsumexp over the masked scores
        sc = torch.einsum("hld,hsd->hls", qt, kt) * h["softmax_scale"]
        sc = sc.masked_fill(~mask, float("-inf"))
        ref_lse = torch.logsumexp(sc, dim=-1).permute(1, 0).numpy()
        assert np.allclose(lse[t0:t1], ref_lse, rtol=1e-6, atol=1e-6)


# ------------------------------------------------------------ closed forms


def test_single_visible_key_returns_its_value_row():
    # Window 1: every query sees exactly one key, itself.
    S = np.array([1, 17, 40, 33])
    L = np.array([1, 5, 40, 1])
    b = W.build_batch("single", 7, S, L, 8, 2, layer_windows=(1,))
    h = W.host_inputs(b)
    out, lse = _run_oracle(h)
    g = 4
    for r in range(len(S)):
        for i in range(int(L[r])):
            t = int(h["query_start_loc"][r]) + i
            pos = int(S[r]) - int(L[r]) + i
            page = h["block_table"][r, pos // 16]
            for hq in range(8):
                vrow = h["v_cache"][page, hq // g, pos % 16]
                assert np.array_equal(out[t, hq], vrow)
                kq = np.dot(brute.bits_to_f64(h["q"][t, hq]), brute.bits_to_f64(h["k_cache"][page, hq // g, pos % 16]))
                assert abs(lse[t, hq] - h["softmax_scale"] * kq) <= 1e-6 * max(1.0, abs(lse[t, hq]))


@pytest.mark.parametrize("window", [0, 7, 64])
def test_zero_query_gives_mean_of_visible_values(window):
    S = np.array([5, 100, 300])
    L = np.array([1, 30, 3])
    b = W.build_batch("zeroq", 8, S, L, 4, 1, layer_windows=(window,))
    h = W.host_inputs(b)
    h["q"] = np.zeros_like(h["q"])
    out, lse = _run_oracle(h)
    vf = brute.bits_to_f64(h["v_cache"])
    for r in range(len(S)):
        for i in range(int(L[r])):
            t = int(h["query_start_loc"][r]) + i
            p = int(S[r]) - int(L[r]) + i
            lo = 0 if window <= 0 else max(0, p - window + 1)
            js = np.arange(lo, p + 1)
            rows = vf[h["block_table"][r, js // 16], 0, js % 16]  # [n, D]
            mean = rows.mean(axis=0)
            o = _f(out[t, 0])
            assert np.all(np.abs(o - mean) <= np.abs(mean) * 2.0**-8 + 1e-30)
            assert abs(lse[t, 0] - math.log(len(js))) <= 1e-6


def test_constant_values_are_reproduced_exactly():
    # Softmax weights sum to one, so a constant value row comes back as is.
    b = W.fuzz_batch(5)
    h = W.host_inputs(b)
    c = torch.tensor([0.7109375], dtype=torch.bfloat16).view(torch.int16).numpy().view(np.uint16)[0]
    h["v_cache"] = np.full_like(h["v_cache"], c)
    out, _ = _run_oracle(h)
    assert np.all(out == c)


def test_two_key_closed_form():
    # q = 8 e0, k0 = 0, k1 = e0 -> scores (0, 1) with scale 1/8; v0 = e0,
    # v1 = e1 -> out = (1, e) / (1 + e) in the first two dims, lse = ln(1 + e).
    D = 64
    one = 0x3F80
    q = np.zeros((1, 1, D), np.uint16)
    q[0, 0, 0] = 0x4100  # 8.0
    kc = np.zeros((1, 1, 16, D), np.uint16)
    vc = np.zeros((1, 1, 16, D), np.uint16)
    kc[0, 0, 1, 0] = one
    vc[0, 0, 0, 0] = one
    vc[0, 0, 1, 1] = one
    out, lse = oracle.paged_attention(q, kc, vc, np.array([[0]], np.int32), np.array([2], np.int32),
                                      np.array([0, 1], np.int32), 0, 0.125)
    e = math.e
    assert out[0, 0, 0] == oracle.double_to_bf16(1 / (1 + e))
    assert out[0, 0, 1] == oracle.double_to_bf16(e / (1 + e))
    assert np.all(out[0, 0, 2:] == 0)
    assert abs(lse[0, 0] - math.log1p(e)) < 1e-6


# ------------------------------------------------------------- invariants


def test_physical_page_relabelling_is_invisible():
    b = W.fuzz_batch(17)
    h = W.host_inputs(b)
    out, lse = _run_oracle(h)
    rng = np.random.default_rng(1)
    P = h["k_cache"].shape[0]
    perm = rng.permutation(P)  # new physical id of old page i is perm[i]
    kc = np.empty_like(h["k_cache"])
    vc = np.empty_like(h["v_cache"])
    kc[perm] = h["k_cache"]
    vc[perm] = h["v_cache"]
    bt = np.where(h["block_table"] >= 0, perm[np.maximum(h["block_table"], 0)], -1).astype(np.int32)
    out2, lse2 = oracle.paged_attention(h["q"], kc, vc, bt, h["seq_lens"], h["query_start_loc"],
                                        h["sliding_window"], h["softmax_scale"])
    assert np.array_equal(out, out2)
    assert np.array_equal(lse, lse2)


def test_paged_equals_unpaged():
    # Same rows laid out contiguously: one page per row, page_size = max S.
    b = W.fuzz_batch(23)
    h = W.host_inputs(b)
    out, lse = _run_oracle(h)
    S = h["seq_lens"]
    Smax = int(S.max())
    B = len(S)
    Hkv, D = h["k_cache"].shape[1], h["k_cache"].shape[3]
    kc = np.zeros((B, Hkv, Smax, D), np.uint16)
    vc = np.zeros((B, Hkv, Smax, D), np.uint16)
    for r in range(B):
        k, v = brute.dense_kv(h["k_cache"], h["v_cache"], h["block_table"][r], int(S[r]), 16)
        pos = np.arange(int(S[r]))
        pages = h["block_table"][r][pos // 16]
        kc[r, :, : S[r]] = h["k_cache"][pages, :, pos % 16].transpose(1, 0, 2)
        vc[r, :, : S[r]] = h["v_cache"][pages, :, pos % 16].transpose(1, 0, 2)
    bt = np.arange(B, dtype=np.int32)[:, None]
    out2, lse2 = oracle.paged_attention(h["q"], kc, vc, bt, S, h["query_start_loc"], h["sliding_window"],
                                        h["softmax_scale"])
    assert np.array_equal(out, out2)
    assert np.array_equal(lse, lse2)


def test_window_wider_than_context_equals_full_context():
    b = W.fuzz_batch(31)
    h = W.host_inputs(b)
    out0, lse0 = _run_oracle(h, window=0)
    big = int(h["seq_lens"].max()) + 1
    out1, lse1 = _run_oracle(h, window=big)
    assert np.array_equal(out0, out1) and np.array_equal(lse0, lse1)


def test_gqa_equals_mha_with_repeated_kv_heads():
    b = W.build_batch("gqa", 9, [50, 130], [20, 1], 8, 2)
    h = W.host_inputs(b)
    out, lse = _run_oracle(h)
    kc = np.repeat(h["k_cache"], 4, axis=1)
    vc = np.repeat(h["v_cache"], 4, axis=1)
    out2, lse2 = oracle.paged_attention(h["q"], kc, vc, h["block_table"], h["seq_lens"], h["query_start_loc"],
                                        0, h["softmax_scale"])
    assert np.array_equal(out, out2) and np.array_equal(lse, lse2)


@pytest.mark.parametrize("window", [0, 24])
def test_causal_and_window_locality(window):
    # Changing keys/values a query may not see leaves its output unchanged;
    # changing the newest key it does see changes it.
    S, L = 90, 40
    b = W.build_batch("causal", 12, [S], [L], 4, 1, layer_windows=(window,))
    h = W.host_inputs(b)
    out, lse = _run_oracle(h)
    i = 17
    p = S - L + i
    lo = 0 if window <= 0 else p - window + 1
    bt = h["block_table"][0]
    kc, vc = h["k_cache"].copy(), h["v_cache"].copy()
    for j in list(range(p + 1, S)) + list(range(0, lo)):
        if bt[j // 16] < 0:
            continue  # page not allocated: nobody may read it
        kc[bt[j // 16], 0, j % 16] ^= 0x0100
        vc[bt[j // 16], 0, j % 16] ^= 0x0100
    out2, lse2 = oracle.paged_attention(h["q"], kc, vc, h["block_table"], h["seq_lens"], h["query_start_loc"],
                                        window, h["softmax_scale"])
    assert np.array_equal(out[i], out2[i]) and np.array_equal(lse[i], lse2[i])
    assert not np.array_equal(out[i + 1:], out2[i + 1:])  # later queries do see them
    vc2 = h["v_cache"].copy()
    vc2[bt[p // 16], 0, p % 16] ^= 0x4000
    out3, _ = oracle.paged_attention(h["q"], h["k_cache"], vc2, h["block_table"], h["seq_lens"],
                                     h["query_start_loc"], window, h["softmax_scale"])
    assert not np.array_equal(out[i], out3[i])


def test_split_keys_merge_by_log_sum_exp():
    # Keys [0, a) and [a, S) of a decode row, attended separately (the second
    # through a window of S - a), merged by lse = logaddexp(lse1, lse2) and
    # out = sum_i exp(lse_i - lse) o_i, equal attention over all S keys.
    S = np.array([200, 77, 1000])
    b = W.build_batch("split", 13, S, [1, 1, 1], 8, 2)
    h = W.host_inputs(b)
    out, lse = _run_oracle(h)
    for r, a in [(0, 64), (1, 1), (2, 999), (2, 333)]:
        sub = {k: v for k, v in h.items()}
        idx = [r]
        q = h["q"][idx]
        bt = h["block_table"][idx]
        qsl = np.array([0, 1], np.int32)
        o1, l1 = oracle.paged_attention(q, h["k_cache"], h["v_cache"], bt, np.array([a], np.int32), qsl, 0,
                                        h["softmax_scale"])
        o2, l2 = oracle.paged_attention(q, h["k_cache"], h["v_cache"], bt, np.array([S[r]], np.int32), qsl,
                                        int(S[r] - a), h["softmax_scale"])
        lm = np.logaddexp(l1.astype(np.float64), l2.astype(np.float64))
        assert np.allclose(lm, lse[r], rtol=0, atol=2e-6)
        om = np.exp(l1 - lm)[..., None] * _f(o1) + np.exp(l2 - lm)[..., None] * _f(o2)
        ref = _f(out[r])
        tol = 2.0**-7 * np.max(np.abs(ref)) + 1e-6  # both partials were rounded to bf16
        assert np.max(np.abs(om[0] - ref)) <= tol


def test_sampled_evaluation_equals_full_evaluation():
    b = W.fuzz_batch(37)
    h = W.host_inputs(b)
    out, lse = _run_oracle(h)
    rng = np.random.default_rng(3)
    tok = rng.integers(0, b.total_q, size=50)
    hd = rng.integers(0, b.num_q_heads, size=50).astype(np.int32)
    so, sl = oracle.paged_attention_sampled(h["q"], h["k_cache"], h["v_cache"], h["block_table"], h["seq_lens"],
                                            h["query_start_loc"], h["sliding_window"], h["softmax_scale"], tok, hd)
    assert np.array_equal(so, out[tok, hd])
    assert np.array_equal(sl, lse[tok, hd])


# --------------------------------------------------------------- kv append


@pytest.mark.parametrize("seed", range(10))
def test_kv_append_bit_exact_against_numpy_scatter(seed):
    b = W.fuzz_batch(seed)
    h = W.host_inputs(b)
    kc, vc = oracle.kv_append(h["k_new"], h["v_new"], h["k_cache"], h["v_cache"], h["block_table"],
                              h["seq_lens"], h["query_start_loc"])
    kb, vb = brute.kv_append(h["k_new"], h["v_new"], h["k_cache"], h["v_cache"], h["block_table"],
                             h["seq_lens"], h["query_start_loc"])
    assert np.array_equal(kc, kb) and np.array_equal(vc, vb)
    # every slot outside [S - L, S) of every row is untouched
    touched = np.zeros(kc.shape[:1] + kc.shape[2:3], bool)
    for r in range(b.num_seqs):
        S, L = int(h["seq_lens"][r]), int(b.q_lens[r])
        for pos in range(S - L, S):
            touched[h["block_table"][r, pos // 16], pos % 16] = True
    same = np.all(kc == h["k_cache"], axis=(1, 3)) & np.all(vc == h["v_cache"], axis=(1, 3))
    assert np.all(same[~touched])


def test_kv_append_never_writes_shared_prompt_pages():
    rng = np.random.default_rng(77)
    grp = np.repeat(np.arange(3), 4)
    prompt = rng.integers(100, 400, size=3)[grp]
    L = np.where(rng.random(12) < 0.5, 1, rng.integers(2, 50, size=12))
    S = prompt + rng.integers(0, 300, size=12) + L
    shared = prompt // 16
    b = W.build_batch("grp", 77, S, L, 8, 2, shared_prefix_pages=shared, prompt_lens=prompt, group_of_row=grp)
    h = W.host_inputs(b)
    kc, vc = oracle.kv_append(h["k_new"], h["v_new"], h["k_cache"], h["v_cache"], h["block_table"],
                              h["seq_lens"], h["query_start_loc"])
    for r in range(b.num_seqs):
        for lp in range(int(shared[r])):
            pg = h["block_table"][r, lp]
            assert np.array_equal(kc[pg], h["k_cache"][pg]) and np.array_equal(vc[pg], h["v_cache"][pg])
    # and members of a group really do share those physical pages
    for g in range(3):
        rows = np.nonzero(grp == g)[0]
        n = int(shared[rows[0]])
        assert n > 0
        assert all(np.array_equal(h["block_table"][rows[0], :n], h["block_table"][r, :n]) for r in rows)


# ------------------------------------------------------------ input checks


def test_oracle_rejects_bad_inputs():
    b = W.config_tiny()
    h = W.host_inputs(b)
    bad = h["seq_lens"].copy()
    bad[0] = 0  # L = 1 > S = 0
    with pytest.raises(oracle.OracleError):
        oracle.paged_attention(h["q"], h["k_cache"], h["v_cache"], h["block_table"], bad, h["query_start_loc"], 0,
                               0.125)
    bt = h["block_table"].copy()
    bt[1, 0] = 9999
    with pytest.raises(oracle.OracleError):
        oracle.paged_attention(h["q"], h["k_cache"], h["v_cache"], bt, h["seq_lens"], h["query_start_loc"], 0, 0.125)
    # the append of row 1 (S = 64, L = 1) writes position 63: logical page 3 only
    oracle.kv_append(h["k_new"], h["v_new"], h["k_cache"], h["v_cache"], bt, h["seq_lens"], h["query_start_loc"])
    bt[1, 3] = -1
    with pytest.raises(oracle.OracleError):
        oracle.kv_append(h["k_new"], h["v_new"], h["k_cache"], h["v_cache"], bt, h["seq_lens"],
                         h["query_start_loc"])


def test_unallocated_pages_outside_the_window_are_never_read():
    b = W.build_batch("swa", 21, [400, 260], [1, 30], 8, 2, layer_windows=(32,))
    h = W.host_inputs(b)
    assert np.any(h["block_table"] == -1)
    out, lse = _run_oracle(h)
    assert np.all(np.isfinite(lse))


# ------------------------------------------------------- attention sinks


def _sinks(hq, seed):
    return np.random.default_rng(seed).normal(0.0, 1.5, size=hq).astype(np.float32)


def test_sinks_at_minus_infinity_change_nothing():
    b = W.fuzz_batch(21)
    h = W.host_inputs(b)
    out, lse = _run_oracle(h)
    out_s, lse_s = oracle.paged_attention(h["q"], h["k_cache"], h["v_cache"], h["block_table"], h["seq_lens"],
                                          h["query_start_loc"], h["sliding_window"], h["softmax_scale"],
                                          sinks=np.full(b.num_q_heads, -np.inf, np.float32))
    assert np.array_equal(out, out_s) and np.array_equal(lse, lse_s)


@pytest.mark.parametrize("sigma,frac", [(0.0, 0.5), (math.log(3.0), 0.25), (-math.log(3.0), 0.75)])
def test_sink_with_one_visible_key_closed_form(sigma, frac):
    # q = 0 and window 1: one key with score 0; the sink adds e^sigma to the
    # normaliser, so out = v / (1 + e^sigma) and lse = ln(1 + e^sigma).
    b = W.build_batch("sink1", 31, [9, 40], [1, 3], 4, 2, layer_windows=(1,))
    h = W.host_inputs(b)
    h["q"] = np.zeros_like(h["q"])
    kc, vc = oracle.kv_append(h["k_new"], h["v_new"], h["k_cache"], h["v_cache"], h["block_table"],
                              h["seq_lens"], h["query_start_loc"])
    out, lse = oracle.paged_attention(h["q"], kc, vc, h["block_table"], h["seq_lens"], h["query_start_loc"], 1,
                                      h["softmax_scale"], sinks=np.full(4, sigma, np.float32))
    vals = brute.bits_to_f64(h["v_new"])  # the query's own key is its new row
    for t in range(out.shape[0]):
        for hq in range(4):
            want = vals[t, hq // 2] * frac
            assert np.all(np.abs(_f(out[t, hq]) - want) <= np.abs(want) * 2.0**-8)
            assert abs(lse[t, hq] - math.log1p(math.exp(np.float32(sigma)))) <= 1e-6


@pytest.mark.parametrize("seed", range(6))
def test_sinks_match_brute_force(seed):
    b = W.fuzz_batch(300 + seed)
    h = W.host_inputs(b)
    kc, vc = oracle.kv_append(h["k_new"], h["v_new"], h["k_cache"], h["v_cache"], h["block_table"],
                              h["seq_lens"], h["query_start_loc"])
    sk = _sinks(b.num_q_heads, seed)
    out, lse = oracle.paged_attention(h["q"], kc, vc, h["block_table"], h["seq_lens"], h["query_start_loc"],
                                      h["sliding_window"], h["softmax_scale"], sinks=sk)
    ref_out, ref_lse = brute.attention(h["q"], kc, vc, h["block_table"], h["seq_lens"], h["query_start_loc"],
                                       h["sliding_window"], h["softmax_scale"], sinks=sk)
    _assert_close_to_exact(out, lse, ref_out, ref_lse)


def test_sink_rescales_the_sinkless_result():
    # Z' = Z + e^sigma: lse' = logaddexp(lse, sigma) and out' = out * e^(lse - lse')
    b = W.fuzz_batch(44)
    h = W.host_inputs(b)
    sk = _sinks(b.num_q_heads, 7)
    out, lse = _run_oracle(h)
    out_s, lse_s = oracle.paged_attention(h["q"], h["k_cache"], h["v_cache"], h["block_table"], h["seq_lens"],
                                          h["query_start_loc"], h["sliding_window"], h["softmax_scale"], sinks=sk)
    want_lse = np.logaddexp(lse.astype(np.float64), sk[None, :].astype(np.float64))
    assert np.allclose(lse_s, want_lse, rtol=0, atol=2e-6 * np.maximum(1, np.abs(want_lse)).max())
    want = _f(out) * np.exp(lse.astype(np.float64) - want_lse)[..., None]
    assert np.all(np.abs(_f(out_s) - want) <= np.abs(want) * 2.0**-7 + 1e-30)


def test_sampled_evaluation_with_sinks_equals_full_evaluation():
    b = W.fuzz_batch(45)
    h = W.host_inputs(b)
    sk = _sinks(b.num_q_heads, 9)
    out, lse = oracle.paged_attention(h["q"], h["k_cache"], h["v_cache"], h["block_table"], h["seq_lens"],
                                      h["query_start_loc"], h["sliding_window"], h["softmax_scale"], sinks=sk)
    rng = np.random.default_rng(3)
    toks = rng.integers(0, out.shape[0], size=20).astype(np.int64)
    heads = rng.integers(0, b.num_q_heads, size=20).astype(np.int32)
    so, sl = oracle.paged_attention_sampled(h["q"], h["k_cache"], h["v_cache"], h["block_table"], h["seq_lens"],
                                            h["query_start_loc"], h["sliding_window"], h["softmax_scale"], toks,
                                            heads, sinks=sk)
    assert np.array_equal(so, out[toks, heads]) and np.array_equal(sl, lse[toks, heads])


# ------------------------------------------------------ rotary embedding


def _rand_bits(shape, seed):
    x = torch.randn(shape, generator=torch.Generator().manual_seed(seed), dtype=torch.bfloat16)
    return x.view(torch.int16).numpy().view(np.uint16).copy()


def test_rope_with_the_identity_table_changes_nothing():
    x = _rand_bits((5, 3, 64), 1)
    tab = np.concatenate([np.ones((10, 32)), np.zeros((10, 32))], axis=1).astype(np.float32)
    assert np.array_equal(oracle.rope(x, np.array([0, 3, 9, 4, 4]), tab), x)


def test_rope_quarter_turn_swaps_halves():
    x = _rand_bits((4, 2, 64), 2)
    tab = np.concatenate([np.zeros((8, 32)), np.ones((8, 32))], axis=1).astype(np.float32)
    y = oracle.rope(x, np.array([1, 2, 3, 7]), tab)
    assert np.array_equal(y[..., 32:], x[..., :32])
    neg = (x[..., 32:] ^ 0x8000).astype(np.uint16)  # -x, exact
    assert np.array_equal(y[..., :32], neg)


def test_rope_of_unit_vectors_gives_the_table_entries():
    tab = W.rope_table(50)
    x = np.zeros((32, 1, 64), np.uint16)
    for i in range(32):
        x[i, 0, i] = 0x3F80  # e_i
    pos = np.arange(32) + 11
    y = _f(oracle.rope(x, pos, tab))
    for i in range(32):
        c, s = float(tab[pos[i], i]), float(tab[pos[i], 32 + i])
        assert y[i, 0, i] == _f(np.array([oracle.double_to_bf16(c)]))[0]
        assert y[i, 0, 32 + i] == _f(np.array([oracle.double_to_bf16(s)]))[0]
        assert np.count_nonzero(y[i, 0]) <= 2


def test_rope_scores_depend_on_relative_position_only():
    tab = W.rope_table(4096)
    q = _rand_bits((1, 8, 64), 3)
    k = _rand_bits((1, 8, 64), 4)
    base = None
    for shift in (0, 7, 300, 3000):
        qr = _f(oracle.rope(q, np.array([40 + shift]), tab))
        kr = _f(oracle.rope(k, np.array([5 + shift]), tab))
        s = (qr * kr).sum(axis=-1)[0]
        bound = 2.0**-7 * (np.linalg.norm(_f(q), axis=-1) * np.linalg.norm(_f(k), axis=-1))[0]
        if base is None:
            base = s
        else:
            assert np.all(np.abs(s - base) <= bound)


def test_rope_preserves_norms():
    tab = W.rope_table(1000)
    x = _rand_bits((16, 4, 64), 5)
    y = oracle.rope(x, np.arange(16) * 61, tab)
    nx, ny = np.linalg.norm(_f(x), axis=-1), np.linalg.norm(_f(y), axis=-1)
    assert np.all(np.abs(nx - ny) <= 2.0**-8 * nx)


def test_token_positions():
    pos = oracle.token_positions([10, 4, 7], [0, 1, 1, 4])
    assert list(pos) == [9, 4, 5, 6]


# ------------------------------------------------------------ fp8 KV pages


def _torch_e4m3(xs):
    """torch's float32 -> float8_e4m3fn conversion (round to nearest even)."""
    t = torch.from_numpy(np.asarray(xs, np.float32)).to(torch.float8_e4m3fn)
    return t.view(torch.uint8).numpy()


def test_e4m3_decoding_matches_torch_for_all_codes():
    codes = np.arange(256, dtype=np.uint8)
    ref = torch.from_numpy(codes).view(torch.float8_e4m3fn).float().numpy().astype(np.float64)
    got = np.array([oracle.e4m3_to_float(c) for c in codes])
    nan = np.isnan(ref)
    assert np.array_equal(nan, np.isnan(got)) and np.array_equal(np.nonzero(nan)[0], [0x7F, 0xFF])
    assert np.array_equal(got[~nan], ref[~nan])
    # format facts: largest 448, smallest subnormal 2^-9, smallest normal 2^-6
    assert got[0x7E] == 448.0 and got[0x01] == 2.0**-9 and got[0x08] == 2.0**-6 and got[0xFE] == -448.0


def test_e4m3_encoding_round_trips_every_code():
    for c in range(256):
        if c & 0x7F == 0x7F:
            continue
        assert oracle.float_to_e4m3(oracle.e4m3_to_float(c)) == c


def test_e4m3_encoding_matches_torch_in_range():
    rng = np.random.default_rng(21)
    mags = np.concatenate([
        rng.uniform(0, 464, 3000),
        np.exp2(rng.uniform(-14, 9, 3000)),
        rng.uniform(0, 2.0**-6, 1000),  # subnormal range
    ])
    mags = mags[mags <= 464]
    xs = (mags * rng.choice([-1.0, 1.0], mags.size)).astype(np.float32)
    got = np.array([oracle.float_to_e4m3(float(x)) for x in xs], np.uint8)
    assert np.array_equal(got, _torch_e4m3(xs))


def test_e4m3_encoding_ties_go_to_the_even_code():
    vals = np.array([oracle.e4m3_to_float(c) for c in range(0x7F)])
    mids = ((vals[:-1] + vals[1:]) / 2).astype(np.float32)  # exact in float32
    got = np.array([oracle.float_to_e4m3(float(m)) for m in mids], np.uint8)
    lo = np.arange(0x7E, dtype=np.uint8)
    assert np.array_equal(got, np.where(lo % 2 == 0, lo, lo + 1))
    assert np.array_equal(got, _torch_e4m3(mids))


def test_e4m3_encoding_saturates():
    for x in [448.0, 449.0, 464.0, 465.0, 1e6, 3.0e38, math.inf]:
        assert oracle.float_to_e4m3(x) == 0x7E and oracle.float_to_e4m3(-x) == 0xFE
    assert oracle.float_to_e4m3(math.nan) & 0x7F == 0x7F
    assert oracle.float_to_e4m3(2.0**-11) == 0 and oracle.float_to_e4m3(-0.0) == 0x80


def _fp8_pools(num_pages, hkv, page, d):
    return (np.zeros((num_pages, hkv, page, d), np.uint8), np.zeros((num_pages, hkv, page, d), np.uint8),
            np.zeros((num_pages, hkv, page), np.float32), np.zeros((num_pages, hkv, page), np.float32))


@pytest.mark.parametrize("seed", range(4))
def test_kv_append_fp8_quantizes_each_row_by_its_absmax(seed):
    b = W.fuzz_batch(500 + seed)
    h = W.host_inputs(b)
    num_pages, hkv, page, d = h["k_cache"].shape
    k8, v8, ks, vs = oracle.kv_append_fp8(h["k_new"], h["v_new"], *_fp8_pools(num_pages, hkv, page, d),
                                          h["block_table"], h["seq_lens"], h["query_start_loc"])
    qsl, sl, bt = h["query_start_loc"], h["seq_lens"], h["block_table"]
    written = np.zeros((num_pages, hkv, page), bool)
    for r in range(len(sl)):
        L, S = int(qsl[r + 1] - qsl[r]), int(sl[r])
        for i in range(L):
            t, pos = int(qsl[r]) + i, S - L + i
            pg, slot = int(bt[r, pos // page]), pos % page
            for kvh in range(hkv):
                written[pg, kvh, slot] = True
                for src, codes, scale in ((h["k_new"], k8, ks), (h["v_new"], v8, vs)):
                    x = oracle.bf16_bits_to_float(src[t, kvh]).astype(np.float32)
                    a = np.float32(np.abs(x).max())
                    if a == 0:
                        assert scale[pg, kvh, slot] == 0 and not codes[pg, kvh, slot].any()
                        continue
                    assert scale[pg, kvh, slot] == a / np.float32(448)
                    want = _torch_e4m3(x * (np.float32(448) / a))
                    assert np.array_equal(codes[pg, kvh, slot], want)
                    assert (want[np.argmax(np.abs(x))] & 0x7F) == 0x7E  # the absmax maps to +-448
                    deq = np.array([oracle.e4m3_to_float(c) for c in want]) * float(scale[pg, kvh, slot])
                    err = np.abs(deq - x.astype(np.float64))
                    # half a quantum: 2^-4 relative for normals, 2^-10 * scale below 2^-6 * scale
                    assert np.all(err <= np.abs(x) * 2.0**-4 * (1 + 1e-6) + float(scale[pg, kvh, slot]) * 2.0**-10)
    assert not k8[~written].any() and not v8[~written].any()
    assert not ks[~written].any() and not vs[~written].any()


def _exact_fp8_batch(seed):
    """A batch whose bf16 pools hold e4m3 values times a power-of-two scale
    per row, so that the fp8 pools describe the very same K and V."""
    b = W.fuzz_batch(seed)
    h = W.host_inputs(b)
    num_pages, hkv, page, d = h["k_cache"].shape
    rng = np.random.default_rng(seed)
    pools = []
    for _ in range(2):
        codes = rng.integers(0, 256, size=(num_pages, hkv, page, d)).astype(np.uint8)
        codes[(codes & 0x7F) == 0x7F] = 0x3A
        scale = np.exp2(rng.integers(-8, -2, size=(num_pages, hkv, page))).astype(np.float32)
        vals = np.array([oracle.e4m3_to_float(c) for c in range(256)])[codes] * scale[..., None]
        bits = torch.from_numpy(vals.astype(np.float32)).to(torch.bfloat16).view(torch.int16).numpy()
        assert np.array_equal(oracle.bf16_bits_to_float(bits.view(np.uint16)), vals)  # exact in bf16
        pools.append((codes, scale, bits.view(np.uint16)))
    return h, pools


@pytest.mark.parametrize("seed", range(4))
def test_fp8_attention_equals_bf16_attention_on_the_same_values(seed):
    h, ((k8, ks, k16), (v8, vs, v16)) = _exact_fp8_batch(600 + seed)
    args = (h["block_table"], h["seq_lens"], h["query_start_loc"], h["sliding_window"], h["softmax_scale"])
    sk = _sinks(h["q"].shape[1], seed) if seed % 2 else None
    o8, l8 = oracle.paged_attention_fp8(h["q"], k8, v8, ks, vs, *args, sinks=sk)
    o16, l16 = oracle.paged_attention(h["q"], k16, v16, *args, sinks=sk)
    assert np.array_equal(o8, o16) and np.array_equal(l8, l16)
    ref_out, ref_lse = brute.attention(h["q"], k16, v16, *args, sinks=sk)
    _assert_close_to_exact(o8, l8, ref_out, ref_lse)


def test_sampled_fp8_evaluation_equals_full_evaluation():
    h, ((k8, ks, _), (v8, vs, _)) = _exact_fp8_batch(610)
    args = (h["block_table"], h["seq_lens"], h["query_start_loc"], h["sliding_window"], h["softmax_scale"])
    out, lse = oracle.paged_attention_fp8(h["q"], k8, v8, ks, vs, *args)
    rng = np.random.default_rng(4)
    toks = rng.integers(0, out.shape[0], size=24).astype(np.int64)
    heads = rng.integers(0, h["q"].shape[1], size=24).astype(np.int32)
    so, sl = oracle.paged_attention_sampled_fp8(h["q"], k8, v8, ks, vs, *args, toks, heads)
    assert np.array_equal(so, out[toks, heads]) and np.array_equal(sl, lse[toks, heads])


def _quantize_pool_oracle(k_bits, v_bits):
    """Whole bf16 pools quantized by the oracle (each page appended as one 16-token row)."""
    P, H, page, D = k_bits.shape
    tok = lambda x: np.ascontiguousarray(x.transpose(0, 2, 1, 3).reshape(P * page, H, D))  # noqa: E731
    z8 = np.zeros((P, H, page, D), np.uint8)
    zs = np.zeros((P, H, page), np.float32)
    return oracle.kv_append_fp8(tok(k_bits), tok(v_bits), z8, z8, zs, zs, np.arange(P, dtype=np.int32)[:, None],
                                np.full(P, page, np.int32), np.arange(P + 1, dtype=np.int32) * page)


@pytest.mark.parametrize("seed", range(3))
def test_fp8_storage_error_stays_within_its_bounds(seed):
    # What the fp8 format changes against bf16 attention on the same inputs:
    # with every score moved by at most delta (sup norm), lse moves by at most
    # delta (log-sum-exp is 1-Lipschitz in the sup norm) and every softmax
    # weight by a factor within e^(+-2 delta), so
    #   |out8 - out16| <= max_j |V8_j - V16_j| + (e^(2 delta) - 1) max_j |V16_j|
    # per output dim, plus the final bf16 rounding of both outputs.
    b = W.fuzz_batch(700 + seed)
    h = W.host_inputs(b)
    kc, vc = oracle.kv_append(h["k_new"], h["v_new"], h["k_cache"], h["v_cache"], h["block_table"],
                              h["seq_lens"], h["query_start_loc"])
    k8, v8, ks, vs = _quantize_pool_oracle(kc, vc)
    args = (h["block_table"], h["seq_lens"], h["query_start_loc"], h["sliding_window"], h["softmax_scale"])
    o16, l16 = oracle.paged_attention(h["q"], kc, vc, *args)
    o8, l8 = oracle.paged_attention_fp8(h["q"], k8, v8, ks, vs, *args)
    val = np.array([oracle.e4m3_to_float(c) for c in range(256)])
    kd, vd = val[k8] * ks[..., None], val[v8] * vs[..., None]  # dequantized pools
    kf, vf = _f(kc), _f(vc)
    q = _f(h["q"])
    g = b.num_q_heads // b.num_kv_heads
    qsl, sl, bt = h["query_start_loc"], h["seq_lens"], h["block_table"]
    checked = 0
    for r in range(len(sl)):
        S, L = int(sl[r]), int(qsl[r + 1] - qsl[r])
        for i in range(L):
            t, pos = int(qsl[r]) + i, S - L + i
            lo = 0 if h["sliding_window"] <= 0 else max(0, pos - h["sliding_window"] + 1)
            js = np.arange(lo, pos + 1)
            pg, sl_ = bt[r, js // 16], js % 16
            for hq in range(b.num_q_heads):
                kv = hq // g
                dk = kd[pg, kv, sl_] - kf[pg, kv, sl_]
                delta = h["softmax_scale"] * np.max(np.abs(dk @ q[t, hq]))
                assert abs(float(l8[t, hq]) - float(l16[t, hq])) <= delta + 1e-5
                dv = np.max(np.abs(vd[pg, kv, sl_] - vf[pg, kv, sl_]), axis=0)
                vmax = np.max(np.abs(vf[pg, kv, sl_]), axis=0)
                bound = dv + np.expm1(2 * delta) * vmax
                ref = _f(o16[t, hq])
                assert np.all(np.abs(_f(o8[t, hq]) - ref) <= bound + 2.0**-8 * (np.abs(ref) + bound) + 1e-30)
                checked += 1
    assert checked > 0
