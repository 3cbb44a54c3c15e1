"""fp8 (e4m3) KV pages through the C ABI: the quantizing append bit for bit
against the oracle, and decode attention over fp8 pages against the
oracle's attention over the same codes, at the parity tolerances."""
import numpy as np
import pytest
import torch

import workloads as W

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    import oracle
    from _gpu import Fp8Run, assert_parity, from_fp8_blocks, oracle_quantize_pool, to_fp8_blocks
    from paper_2608_22167_gb300 import mcpu


def _decode_batch(seed, B=6, lo=1, hi=3000, heads=(64, 8), window=0, **kw):
    rng = np.random.default_rng(seed)
    S = rng.integers(lo, hi, size=B)
    return W.build_batch("fp8", seed, S, np.ones(B, np.int64), heads[0], heads[1], layer_windows=(window,), **kw)


def _check_append(run):
    run.append()
    code, bits = run.status()
    assert code == 0, f"device status bits {bits}"
    k8, v8, ks, vs = run.oracle_append()
    gk8, gv8, gks, gvs = run.pools_host()
    assert np.array_equal(gk8, k8), "k codes differ"
    assert np.array_equal(gv8, v8), "v codes differ"
    assert np.array_equal(gks.view(np.uint32), ks.view(np.uint32)), "k scales differ"
    assert np.array_equal(gvs.view(np.uint32), vs.view(np.uint32)), "v scales differ"
    return k8, v8, ks, vs


def _full_check(batch, flags=0, split_pages=0, sinks=None, garbage_slots=False, what=""):
    run = Fp8Run(batch, garbage_slots=garbage_slots)
    pools = _check_append(run)
    run.forward(flags=flags, split_pages=split_pages, sinks=sinks)
    code, bits = run.status()
    assert code == 0, f"device status bits {bits}"
    h = run.h
    ro, rl = oracle.paged_attention_fp8(h["q"], *pools, h["block_table"], h["seq_lens"], h["query_start_loc"],
                                        h["sliding_window"], h["softmax_scale"], sinks=sinks)
    go, gl = run.out_host()
    return run, assert_parity(go, gl, oracle.bf16_bits_to_float(ro), rl, what or batch.name)


# ------------------------------------------------------------------ append


@pytest.mark.parametrize("seed", range(6))
def test_append_quantizes_bit_exactly(seed):
    # decode and append rows, every row's values scaled by its own power of ten
    rng = np.random.default_rng(seed)
    B = 7
    S = rng.integers(1, 800, size=B)
    L = np.where(rng.random(B) < 0.5, 1, np.minimum(S, rng.integers(1, 120, size=B)))
    b = W.build_batch("fp8app", 90 + seed, S, L, 16, 4)
    lay = b.layers[0]
    T = b.total_q
    mag = torch.from_numpy(10.0 ** rng.uniform(-6, 6, size=(T, 4, 1))).to(torch.bfloat16)
    lay.k_new.mul_(mag)
    lay.v_new.mul_(mag.flip(0))
    lay.k_new[0] = 0  # an all-zero row: zero codes, zero scale
    lay.v_new[-1, 1, :7] = 0
    _check_append(Fp8Run(b))


def test_append_rounding_edges():
    # values that land exactly on e4m3 midpoints, subnormal codes and the
    # largest magnitude in one row
    b = W.build_batch("fp8edge", 5, [40], [40], 8, 2)
    lay = b.layers[0]
    vals = [oracle.e4m3_to_float(c) for c in range(0x7F)]
    mids = [(a + c) / 2 for a, c in zip(vals[:-1], vals[1:])]
    rng = np.random.default_rng(0)
    for t in range(40):
        for h in range(2):
            row = np.array(rng.choice(mids + vals, size=64), np.float64) * rng.choice([-1, 1], size=64)
            row[rng.integers(0, 64)] = 448.0  # absmax 448: inverse scale exactly 1
            x = torch.from_numpy(row).to(torch.bfloat16)
            lay.k_new[t, h] = x
            lay.v_new[t, h] = x * 2.0**-60
    _check_append(Fp8Run(b))


def test_append_reports_bad_pages_and_lengths():
    b = W.build_batch("fp8bad", 6, [50, 70], [1, 20], 8, 2)
    run = Fp8Run(b)
    run.bt[1, 3] = 10**6
    run.append()
    code, bits = run.status()
    assert bits & mcpu.STATUS_BAD_PAGE
    mcpu.mcpu_reset_device_status(run.ws)
    run.sl[0] = 10**6
    run.append()
    code, bits = run.status()
    assert bits & mcpu.STATUS_BAD_LENGTHS


# ----------------------------------------------------------------- forward


def test_tiny_decode_fp8():
    _full_check(W.config_tiny(), what="tiny fp8")


@pytest.mark.parametrize("seed", range(10))
def test_fuzz_decode_batches(seed):
    rng = np.random.default_rng(seed)
    g = int(rng.choice([1, 2, 4, 8]))
    hkv = int(rng.choice([1, 2, 8]))
    b = _decode_batch(300 + seed, B=int(rng.integers(1, 12)), hi=int(rng.choice([40, 600, 4000])),
                      heads=(g * hkv, hkv))
    _full_check(b, what=f"fp8 fuzz{seed}")


@pytest.mark.parametrize("split_pages", [1, 3, 8, 1000])
def test_split_rows(split_pages):
    b = W.build_batch("fp8split", 55, [700, 33, 2049, 16, 1, 5000], np.ones(6, np.int64), 32, 8)
    run, _ = _full_check(b, split_pages=split_pages, what=f"fp8 split{split_pages}")
    if split_pages <= 3:
        assert run.header()["n_merge"] > 0


@pytest.mark.parametrize("window", [1, 16, 128, 1000])
def test_sliding_window(window):
    _full_check(_decode_batch(70 + window, B=8, window=window), what=f"fp8 window{window}")


def _grouped(seed, groups=3, group_size=8):
    rng = np.random.default_rng(seed)
    grp = np.repeat(np.arange(groups), group_size)
    prompt = np.repeat(rng.integers(100, 1500, size=groups), group_size)
    S = prompt + rng.integers(1, 800, size=groups * group_size)
    return W.build_batch("fp8groups", seed, S, np.ones(len(S), np.int64), 64, 8, shared_prefix_pages=prompt // 16,
                         prompt_lens=prompt, group_of_row=grp)


@pytest.mark.parametrize("seed", [1, 2])
def test_cascade_groups(seed):
    b = _grouped(seed)
    run, _ = _full_check(b, what="fp8 cascade")
    assert run.header()["n_cascade"] > 0
    out1, lse1 = run.out_host()
    run.forward(flags=mcpu.FLAG_NO_CASCADE)
    out2, lse2 = run.out_host()
    assert np.max(np.abs(out1 - out2)) <= 2e-2 and np.max(np.abs(lse1 - lse2)) <= 1e-3


@pytest.mark.parametrize("seed", range(3))
def test_sinks(seed):
    rng = np.random.default_rng(seed)
    b = _decode_batch(500 + seed, B=8, hi=2500)
    sk = rng.normal(0, 2, size=b.num_q_heads).astype(np.float32)
    _full_check(b, sinks=sk, split_pages=int(rng.choice([0, 2])), what="fp8 sinks")


def test_sinks_with_cascade_groups():
    b = _grouped(9)
    sk = np.random.default_rng(9).normal(0, 2, size=b.num_q_heads).astype(np.float32)
    _full_check(b, sinks=sk, what="fp8 sinks cascade")


def test_unwritten_slots_may_hold_nan_codes_and_scales():
    b = _decode_batch(61, B=6, hi=900, pool_slack_pages=8)
    _full_check(b, garbage_slots=True, what="fp8 garbage")


def test_wide_value_ranges():
    # K rows scaled by 2^-4 .. 2^2 and V rows by 2^-30 .. 1 within one sequence
    b = _decode_batch(62, B=5, hi=2000)
    pool = b.pools["w0"]
    rng = np.random.default_rng(62)
    P = pool.k_cache.shape[0]
    pool.k_cache.mul_(torch.from_numpy(2.0 ** rng.uniform(-4, 2, size=(P, 1, 16, 1))).to(torch.bfloat16))
    pool.v_cache.mul_(torch.from_numpy(2.0 ** rng.uniform(-30, 0, size=(P, 1, 16, 1))).to(torch.bfloat16))
    _full_check(b, what="fp8 wide ranges")


def test_append_rows_are_refused():
    b = W.build_batch("fp8mixed", 7, [100, 300], [1, 5], 16, 2)
    run = Fp8Run(b)
    with pytest.raises(mcpu.McpuError) as e:
        run.forward()
    assert e.value.code == 2  # MCPU_ERR_UNSUPPORTED, nothing launched
    # same totals as an all-decode batch, but one row appends and one is empty
    b2 = W.build_batch("fp8mixed2", 8, [100, 300, 50], [0, 2, 1], 16, 2)
    run2 = Fp8Run(b2)
    run2.forward()
    code, bits = run2.status()
    assert code == 10 and bits & mcpu.STATUS_UNSUPPORTED_ROW
    # the decode row is still answered
    h = run2.h  # nothing was appended: the pools are the prefilled ones
    ro, rl = oracle.paged_attention_fp8(h["q"][2:3], *run2.before, h["block_table"][2:3], h["seq_lens"][2:3],
                                        np.array([0, 1], np.int32), 0, h["softmax_scale"])
    go, gl = run2.out_host()
    assert_parity(go[2:3], gl[2:3], oracle.bf16_bits_to_float(ro), rl, "decode row beside a skipped append row")


def test_bad_page_is_reported():
    b = _decode_batch(63, B=4, hi=600)
    run = Fp8Run(b)
    run.append()
    run.bt[2, 0] = -5
    run.forward()
    code, bits = run.status()
    assert bits & mcpu.STATUS_BAD_PAGE
    assert np.all(np.isfinite(run.out_host()[0][[0, 1, 3]]))


def test_decode_batch_sampled_at_full_size():
    b = W.config_decode()
    run = Fp8Run(b)
    pools = _check_append(run)
    run.forward()
    assert run.status()[0] == 0
    rng = np.random.default_rng(5)
    h = run.h
    toks = rng.integers(0, b.total_q, size=192).astype(np.int64)
    heads = rng.integers(0, b.num_q_heads, size=192).astype(np.int32)
    ro, rl = oracle.paged_attention_sampled_fp8(h["q"], *pools, h["block_table"], h["seq_lens"],
                                                h["query_start_loc"], 0, h["softmax_scale"], toks, heads)
    go, gl = run.out_host()
    assert_parity(go[toks, heads], gl[toks, heads], oracle.bf16_bits_to_float(ro), rl, "decode_b64 fp8")


def _device_quantized_pool(pool, device="cuda"):
    """An fp8 pool holding every page of a bf16 pool, written on the device by
    mcpu_kv_append_fp8 (each page appended as one 16-token row). Only the
    unchecked rows' pages keep these codes."""
    P, H, page, D = pool.k_cache.shape
    kv8 = mcpu.new_fp8_pool(P, H, device)
    status = torch.zeros(1, dtype=torch.int32, device=device)
    for p0 in range(0, P, 2048):
        n = min(2048, P - p0)
        kn = pool.k_cache[p0:p0 + n].permute(0, 2, 1, 3).reshape(n * page, H, D).contiguous()
        vn = pool.v_cache[p0:p0 + n].permute(0, 2, 1, 3).reshape(n * page, H, D).contiguous()
        bt = torch.arange(p0, p0 + n, dtype=torch.int32, device=device).view(n, 1)
        sl = torch.full((n,), page, dtype=torch.int32, device=device)
        qsl = torch.arange(0, (n + 1) * page, page, dtype=torch.int32, device=device)
        mcpu.mcpu_kv_append_fp8(kn, vn, kv8, bt, sl, qsl, status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    return kv8


def test_long_batch_sampled_at_full_size():
    # the long-horizon batch (512 rows, 33 GB of bf16 KV) over fp8 pages, in
    # the bench's launch configuration. The checked rows' pages hold the
    # oracle's codes; the rest of the pool is quantized on the device.
    b = W.config_long(device="cuda")
    lay = b.layers[0]
    pool = b.pools[lay.pool]
    order = np.argsort(b.seq_lens)
    rows = sorted(set(int(r) for r in list(order[:2]) + list(order[-3:]) + list(order[256:259])))
    h = W.host_rows(b, rows)
    bt_rows = pool.block_table[rows]
    used = np.unique(bt_rows[bt_rows >= 0])  # compact page i of h is physical page used[i]
    before = oracle_quantize_pool(h["k_cache"], h["v_cache"])
    kv8 = _device_quantized_pool(pool)
    used_t = torch.as_tensor(used.astype(np.int64), device="cuda")
    kv8.index_copy_(0, used_t, torch.from_numpy(to_fp8_blocks(*before)).to("cuda"))
    bt = torch.from_numpy(pool.block_table).to("cuda")
    sl = torch.from_numpy(b.seq_lens).to("cuda")
    qsl = torch.from_numpy(b.query_start_loc).to("cuda")
    ws = mcpu.new_workspace(mcpu.dims_fp8(lay.q, kv8, bt, sl), "cuda")
    out = torch.full_like(lay.q, float("nan"))
    lse = torch.full(lay.q.shape[:2], float("nan"), dtype=torch.float32, device="cuda")
    mcpu.mcpu_kv_append_fp8(lay.k_new, lay.v_new, kv8, bt, sl, qsl, mcpu.status_word(ws))
    mcpu.mcpu_paged_attention_forward_fp8(lay.q, kv8, bt, sl, qsl, 0, b.softmax_scale, out, lse, ws)
    code, bits = mcpu.mcpu_read_device_status(ws)
    assert code == 0, f"device status bits {bits}"
    after = oracle.kv_append_fp8(h["k_new"], h["v_new"], *before, h["block_table"], h["seq_lens"],
                                 h["query_start_loc"])
    got = from_fp8_blocks(kv8.index_select(0, used_t).cpu().numpy())
    for g, r, what in zip(got, after, ("k codes", "v codes", "k scales", "v scales")):
        assert np.array_equal(np.ascontiguousarray(g).view(np.uint8), np.ascontiguousarray(r).view(np.uint8)), what
    n_tok = int(h["query_start_loc"][-1])
    toks = np.repeat(np.arange(n_tok, dtype=np.int64), b.num_q_heads)
    heads = np.tile(np.arange(b.num_q_heads, dtype=np.int32), n_tok)
    ro, rl = oracle.paged_attention_sampled_fp8(h["q"], *after, h["block_table"], h["seq_lens"],
                                                h["query_start_loc"], 0, h["softmax_scale"], toks, heads)
    full = h["token_map"][toks]
    go = out.float().cpu().numpy()[full, heads]
    gl = lse.cpu().numpy()[full, heads]
    assert_parity(go, gl, oracle.bf16_bits_to_float(ro), rl, "long_b512 fp8")


@pytest.mark.parametrize("slices", [1, 3])
@pytest.mark.parametrize("seed", range(3))
def test_host_buffer_call(seed, slices):
    # mcpu_paged_attention_host_fp8: q / k_new / v_new / out / lse in host memory
    b = _decode_batch(3700 + seed, B=9, window=(0, 128, 0)[seed])
    run = Fp8Run(b)
    lay = b.layers[0]
    pin = lambda t: t.cpu().contiguous().pin_memory()  # noqa: E731
    qh, knh, vnh = pin(lay.q), pin(lay.k_new), pin(lay.v_new)
    slh = torch.from_numpy(b.seq_lens).to(torch.int32)
    qslh = torch.from_numpy(b.query_start_loc).to(torch.int32)
    out_h = torch.full(qh.shape, float("nan"), dtype=torch.bfloat16).pin_memory()
    lse_h = torch.full(qh.shape[:2], float("nan"), dtype=torch.float32).pin_memory()
    st = mcpu.HostStage(qh.shape[0], b.num_seqs, b.num_q_heads, b.num_kv_heads)
    mcpu.mcpu_paged_attention_host_fp8(st, qh, knh, vnh, run.kv8, run.bt, slh, qslh, run.window, b.softmax_scale,
                                       out_h, lse_h, run.ws, slices=slices)
    mcpu.mcpu_host_stage_sync(st)
    code, bits = run.status()
    assert code == 0, f"device status bits {bits}"
    pools = run.oracle_append()
    for g, r, what in zip(run.pools_host(), pools, ("k codes", "v codes", "k scales", "v scales")):
        assert np.array_equal(np.ascontiguousarray(g).view(np.uint8), np.ascontiguousarray(r).view(np.uint8)), what
    h = run.h
    ro, rl = oracle.paged_attention_fp8(h["q"], *pools, h["block_table"], h["seq_lens"], h["query_start_loc"],
                                        h["sliding_window"], h["softmax_scale"])
    assert_parity(out_h.float().numpy(), lse_h.numpy(), oracle.bf16_bits_to_float(ro), rl, f"host fp8 {seed}")
    st.close()


def test_fp8_and_bf16_paths_agree_on_exactly_representable_pools():
    # pools whose bf16 values are e4m3 codes times power-of-two row scales:
    # both storage formats describe the same K and V
    b = _decode_batch(64, B=6, hi=1500)
    pool = b.pools["w0"]
    rng = np.random.default_rng(64)
    vals = np.array([oracle.e4m3_to_float(c) for c in range(256)])
    for cache in (pool.k_cache, pool.v_cache):
        codes = rng.integers(0, 256, size=tuple(cache.shape)).astype(np.uint8)
        codes[(codes & 0x7F) == 0x7F] = 0x30
        codes[..., 0] = 0x7E  # every row's absmax is 448 * scale: requantizing is exact
        scale = 2.0 ** rng.integers(-12, -8, size=tuple(cache.shape[:3]) + (1,))  # |values| <= 1.75
        cache.copy_(torch.from_numpy(vals[codes] * scale).to(torch.bfloat16))
    lay = b.layers[0]
    for x in (lay.k_new, lay.v_new):
        codes = rng.integers(0, 0x7E, size=tuple(x.shape)).astype(np.uint8)
        codes[..., 0] = 0x7E
        x.copy_(torch.from_numpy(vals[codes] * 2.0**-8).to(torch.bfloat16))
    run8, _ = _full_check(b, what="fp8 exact")
    from _gpu import Run, oracle_full
    run16 = Run(b)
    run16.append()
    run16.forward()
    assert run16.status()[0] == 0
    ref_out, ref_lse, _ = oracle_full(b)  # bf16 oracle: equal to the fp8 oracle on these pools
    o8, l8 = run8.out_host()
    o16, l16 = run16.out_host()
    assert_parity(o16, l16, ref_out, ref_lse, "bf16 path, exact pools")
    assert_parity(o8, l8, o16, l16, "fp8 vs bf16 path")


def test_cuda_graph_replay():
    b = _decode_batch(65, B=16, hi=3000)
    run = Fp8Run(b)
    pools = _check_append(run)
    run.forward()  # first call on the device before capture
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        with torch.cuda.graph(g, stream=s):
            run.forward()
    run.out.fill_(float("nan"))
    g.replay()
    torch.cuda.synchronize()
    assert run.status()[0] == 0
    h = run.h
    ro, rl = oracle.paged_attention_fp8(h["q"], *pools, h["block_table"], h["seq_lens"], h["query_start_loc"], 0,
                                        h["softmax_scale"])
    go, gl = run.out_host()
    assert_parity(go, gl, oracle.bf16_bits_to_float(ro), rl, "fp8 graph replay")


def test_programmatic_launches_match_ordinary_ones_bitwise():
    # fp8 chain on one stream: the planner, the cascade pass (after the
    # decode kernel) and the merge (after the cascade pass) are programmatic
    # launches unless phase events are recorded; both forms, and a graph of
    # the programmatic one, agree bit for bit on groups with split rows
    b = _grouped(7)
    run, _ = _full_check(b, split_pages=2, what="fp8 programmatic")
    assert run.header()["n_cascade"] > 0 and run.header()["n_merge"] > 0
    out_p, lse_p = run.out_host()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(mcpu.NUM_PHASE_EVENTS)]
    for e in ev:  # torch creates the CUDA event at its first record
        e.record()
    run.out.fill_(float("nan"))
    mcpu.mcpu_paged_attention_forward_fp8(run.q, run.kv8, run.bt, run.sl, run.qsl, run.window, b.softmax_scale,
                                          run.out, run.lse, run.ws, split_pages=2, phase_events=ev)
    torch.cuda.synchronize()
    assert run.status()[0] == 0
    out_o, lse_o = run.out_host()
    assert np.array_equal(out_p, out_o) and np.array_equal(lse_p, lse_o)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        run.forward(split_pages=2)
    run.out.fill_(float("nan"))
    g.replay()
    torch.cuda.synchronize()
    assert run.status()[0] == 0
    out_g, lse_g = run.out_host()
    assert np.array_equal(out_p, out_g) and np.array_equal(lse_p, lse_g)
