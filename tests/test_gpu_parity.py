"""GPU parity: the CUDA path through the C ABI against the CPU oracle on the
same seeded inputs, element by element on small batches and on sampled
outputs at the full workload sizes. KV append is compared bit for bit."""
import numpy as np
import pytest
import torch

import workloads as W

pytestmark = pytest.mark.gpu

import oracle

if torch.cuda.is_available():
    from _gpu import Run, assert_parity, oracle_full, oracle_sampled
    from paper_2608_22167_gb300 import mcpu


def _poison_unseen_slots(batch, layer=0):
    """Writes NaN into every K and V slot of the layer's pool that no query of
    the batch can see (slots past a row's end on its last page, slots before
    a window on its first page, the pool's spare pages), as memory that was
    never written may hold. The oracle reads visible keys only."""
    lay = batch.layers[layer]
    pool = batch.pools[lay.pool]
    P = pool.k_cache.shape[0]
    seen = np.zeros((P, 16), bool)
    bt, S, L = pool.block_table, batch.seq_lens, batch.q_lens
    W_ = lay.sliding_window
    for r in range(batch.num_seqs):
        if L[r] == 0:
            continue
        lo = 0 if W_ <= 0 else max(0, int(S[r] - L[r]) - W_ + 1)
        j = np.arange(lo, int(S[r]))
        seen[bt[r, j // 16], j % 16] = True
    hide = torch.from_numpy(~seen)
    for t in (pool.k_cache, pool.v_cache):
        t.permute(0, 2, 1, 3)[hide.to(t.device)] = float("nan")
    return int((~seen).sum())


def _full_check(batch, layer=0, flags=0, split_pages=0, what="", sinks=None):
    run = Run(batch, layer)
    run.append()
    run.forward(flags=flags, split_pages=split_pages, sinks=sinks)
    code, bits = run.status()
    assert code == 0, f"device status bits {bits}"
    ref_out, ref_lse, (okc, ovc) = oracle_full(batch, layer, sinks=sinks)
    assert np.array_equal(W.to_host(run.kc), okc), "k pool differs after append"
    assert np.array_equal(W.to_host(run.vc), ovc), "v pool differs after append"
    got_out, got_lse = run.out_host()
    return run, assert_parity(got_out, got_lse, ref_out, ref_lse, what or batch.name)


def test_tiny_decode():
    _full_check(W.config_tiny())


@pytest.mark.parametrize("seed", range(24))
def test_fuzz_small_batches(seed):
    _full_check(W.fuzz_batch(seed), what=f"fuzz{seed}")


@pytest.mark.parametrize("seed", range(6))
def test_fuzz_long_rows(seed):
    # a few rows long enough for many splits and several append tiles
    _full_check(W.fuzz_batch(1000 + seed, max_len=3000, max_chunk=300), what=f"fuzzlong{seed}")


@pytest.mark.parametrize("seed", range(4))
def test_peaked_inputs(seed):
    rng = np.random.default_rng(200 + seed)
    B = int(rng.integers(2, 7))
    S = rng.integers(20, 1500, size=B)
    L = np.where(rng.random(B) < 0.5, 1, np.minimum(S, rng.integers(2, 200, size=B)))
    b = W.build_batch("peaked", 300 + seed, S, L, 64, 8, layer_windows=(int(rng.choice([0, 128])),), peaked=True)
    _full_check(b, what=f"peaked{seed}")


@pytest.mark.parametrize("seed", range(6))
def test_append_kernels_agree(seed):
    # the tcgen05 append kernel (default) and the mma.sync one, both vs the oracle
    rng = np.random.default_rng(400 + seed)
    B = int(rng.integers(1, 6))
    S = rng.integers(2, 3000, size=B)
    L = np.minimum(S, rng.integers(2, 400, size=B))
    g = int(rng.choice([1, 2, 4, 8]))
    W_ = int(rng.choice([0, 0, 128, 37]))
    b = W.build_batch("appends", 600 + seed, S, L, 2 * g, 2, layer_windows=(W_,))
    run, _ = _full_check(b, what="tcgen05 append")
    tc_out, tc_lse = run.out_host()
    run2, _ = _full_check(b, flags=mcpu.FLAG_MMA_SYNC_APPEND, what="mma.sync append")
    ms_out, ms_lse = run2.out_host()
    assert np.max(np.abs(tc_out - ms_out)) <= 2e-2
    assert np.max(np.abs(tc_lse - ms_lse)) <= 1e-3


@pytest.mark.parametrize("window", [0, 128])
def test_many_append_tiles_per_cta(window):
    # thousands of append tiles: every persistent CTA runs many items in a row
    rng = np.random.default_rng(700 + window)
    B = 64
    L = rng.integers(200, 400, size=B)
    S = L + rng.integers(0, 900, size=B)
    b = W.build_batch("manytiles", 800 + window, S, L, 64, 8, layer_windows=(window,))
    run, _ = _full_check(b, what=f"manytiles w{window}")
    assert run.header()["n_append"] * 8 > 20 * 152


def test_side_stream_and_serial_orders_agree_bitwise():
    # decode kernels on the library's side stream (default) or all on one stream
    rng = np.random.default_rng(41)
    S = rng.integers(1, 5000, size=20)
    L = np.where(np.arange(20) % 4 == 0, np.minimum(S, rng.integers(2, 300, size=20)), 1)
    b = W.build_batch("sides", 42, S, L, 64, 8)
    run, _ = _full_check(b, what="side stream")
    out1, lse1 = run.out_host()
    run.forward(flags=mcpu.FLAG_SERIAL)
    assert run.status()[0] == 0
    out2, lse2 = run.out_host()
    assert np.array_equal(out1, out2) and np.array_equal(lse1, lse2)


@pytest.mark.parametrize("split_pages", [1, 2, 3, 8, 1000])
def test_split_length_does_not_change_results(split_pages):
    b = W.build_batch("splits", 55, [700, 33, 2049, 16, 1], [1, 1, 1, 1, 1], 32, 8)
    run, _ = _full_check(b, split_pages=split_pages, what=f"split{split_pages}")
    hdr = run.header()
    if split_pages <= 3:
        assert hdr["n_merge"] > 0 and hdr["n_decode"] > b.num_seqs


@pytest.mark.parametrize("window", [1, 16, 128, 1000])
def test_sliding_window(window):
    rng = np.random.default_rng(window)
    B = 6
    S = rng.integers(1, 2500, size=B)
    L = np.where(np.arange(B) % 2 == 0, 1, np.minimum(S, rng.integers(2, 300, size=B)))
    b = W.build_batch("win", 77 + window, S, L, 64, 8, layer_windows=(window,))
    _full_check(b, what=f"window{window}")


def _grouped_batch(seed, groups=3, group_size=8, append_frac=0.25):
    rng = np.random.default_rng(seed)
    grp = np.repeat(np.arange(groups), group_size)
    prompt = rng.integers(100, 1200, size=groups)[grp]
    B = groups * group_size
    L = np.where(rng.random(B) < append_frac, rng.integers(2, 100, size=B), 1)
    S = prompt + rng.integers(0, 600, size=B) + L
    shared = prompt // 16
    return W.build_batch(f"groups{seed}", seed, S, L, 64, 8, shared_prefix_pages=shared, prompt_lens=prompt,
                         group_of_row=grp)


@pytest.mark.parametrize("seed", [1, 2, 3])
def test_cascade_matches_oracle_and_flat(seed):
    b = _grouped_batch(seed)
    run, _ = _full_check(b, what="cascade")
    hdr = run.header()
    assert hdr["n_cascade"] > 0, "shared prompt pages were not detected"
    casc_out, casc_lse = run.out_host()
    run2, _ = _full_check(b, flags=mcpu.FLAG_NO_CASCADE, what="flat")
    assert run2.header()["n_cascade"] == 0
    flat_out, flat_lse = run2.out_host()
    assert np.max(np.abs(casc_out - flat_out)) <= 2e-2
    assert np.max(np.abs(casc_lse - flat_lse)) <= 1e-3


def test_groups_larger_than_a_cascade_item():
    # 13 decode members in one group: split into balanced subgroups
    b = _grouped_batch(9, groups=2, group_size=13, append_frac=0.0)
    run, _ = _full_check(b, what="biggroup")
    assert run.header()["n_cascade"] >= 2


def _ws_lcp_offset(B, T, g):
    """Byte offset of the per-row shared-prefix array in the workspace (the
    C ABI's workspace layout: header, decode, cascade, member, append and
    merge records, each array 256-byte aligned)."""
    al = lambda x: (x + 255) // 256 * 256  # noqa: E731
    off = 256
    off = al(off + 32 * (B + 4096 + 1))
    off = al(off + 32 * (B // 2 + 4096 + 1))
    off = al(off + 16 * (B + 1))
    off = al(off + 32 * (T // (64 // g) + B + 1))
    off = al(off + 16 * (B + 1))
    return off


def test_long_shared_prefixes_are_measured_exactly():
    # prompts of 562, 1025 and 1312 full pages: the prefix scan (512 page
    # ids per step) ends in its first, second and third step; adjacent
    # groups differ at page 0
    rng = np.random.default_rng(77)
    groups, gs = 3, 4
    grp = np.repeat(np.arange(groups), gs)
    prompt = np.array([9000, 16400, 21000])[grp]
    S = prompt + rng.integers(1, 300, size=groups * gs)
    b = W.build_batch("longprefix", 78, S, np.ones(len(S), np.int64), 64, 8, shared_prefix_pages=prompt // 16,
                      prompt_lens=prompt, group_of_row=grp)
    run, _ = _full_check(b, what="long prefixes")
    assert run.header()["n_cascade"] > 0
    B = b.num_seqs
    off = _ws_lcp_offset(B, b.total_q, b.num_q_heads // b.num_kv_heads)
    lcp = run.ws[off:off + 4 * B].view(torch.int32).cpu().numpy()
    want = np.array([0] + [int(prompt[r]) // 16 if grp[r] == grp[r - 1] else 0 for r in range(1, B)])
    assert np.array_equal(lcp, want), (lcp, want)


def test_rows_without_queries_and_single_key_rows():
    b = W.build_batch("edge", 91, [1, 5, 16, 17, 40], [1, 0, 16, 0, 3], 16, 2)
    run, _ = _full_check(b, what="edge")


@pytest.mark.parametrize("group", [1, 2, 4, 8])
def test_gqa_ratios(group):
    b = W.build_batch(f"g{group}", 31 + group, [300, 77, 1200], [1, 50, 1], 2 * group, 2)
    _full_check(b, what=f"gqa{group}")


@pytest.mark.parametrize("case", ["decode", "split", "window", "append", "append_window", "mma_sync", "cascade"])
def test_unwritten_slots_may_hold_nan(case):
    # Slots no query can see hold NaN in K and V (never-written memory may):
    # the kernels mask their scores and zero their V rows, since a zero
    # weight does not cancel NaN. Every output must match the oracle, which
    # reads visible keys only.
    rng = np.random.default_rng(len(case) * 31 + ord(case[0]))
    flags, split = 0, 0
    if case == "cascade":
        b = _grouped_batch(17)
    else:
        B = 7
        S = rng.integers(20, 1500, size=B)
        S[0] = 16 * 37 + 5  # a partial last page
        app = case.startswith("append") or case == "mma_sync"
        L = np.where((np.arange(B) % 2 == 0) & app, np.minimum(S, rng.integers(2, 300, size=B)), 1)
        win = 100 if case.endswith("window") or case == "window" else 0
        b = W.build_batch(f"nan_{case}", 500 + len(case), S, L, 64, 8, layer_windows=(win,), pool_slack_pages=5)
        flags = mcpu.FLAG_MMA_SYNC_APPEND if case == "mma_sync" else 0
        split = 2 if case == "split" else 0
    assert _poison_unseen_slots(b) > 0
    run, _ = _full_check(b, flags=flags, split_pages=split, what=f"NaN in unseen slots ({case})")
    if case == "cascade":
        assert run.header()["n_cascade"] > 0
    if case == "split":
        assert run.header()["n_merge"] > 0


# ---------------------------------------------------------------- full sizes


def _appended_pages_bitexact(batch, run, layer=0):
    """Every page this step's KV append wrote (all rows: one slot per decode
    row, the whole chunk of an append row), compared bit for bit with the
    oracle's KV append of those rows: the touched pages are gathered before
    (from the batch, which the run does not modify) and after the append,
    into a compact pool with a renumbered block table."""
    lay = batch.layers[layer]
    pool = batch.pools[lay.pool]
    S, L, qsl = batch.seq_lens.astype(np.int64), batch.q_lens.astype(np.int64), batch.query_start_loc
    rows = np.nonzero(L > 0)[0]
    bt = pool.block_table
    touched = np.unique(np.concatenate([bt[r, (S[r] - L[r]) // 16:(S[r] - 1) // 16 + 1] for r in rows]))
    assert np.all(touched >= 0)
    remap = np.full(pool.num_pages, -1, np.int64)
    remap[touched] = np.arange(touched.shape[0])
    bt_c = np.full((len(rows), bt.shape[1]), -1, np.int32)
    for i, r in enumerate(rows):
        lp = np.arange((S[r] - L[r]) // 16, (S[r] - 1) // 16 + 1)
        bt_c[i, lp] = remap[bt[r, lp]]
    idx = torch.as_tensor(touched, device=pool.k_cache.device)
    tok = torch.as_tensor(np.concatenate([np.arange(qsl[r], qsl[r + 1]) for r in rows]), device=lay.k_new.device)
    qsl_c = np.zeros(len(rows) + 1, np.int32)
    qsl_c[1:] = np.cumsum(L[rows])
    want_k, want_v = oracle.kv_append(W.to_host(lay.k_new.index_select(0, tok)),
                                      W.to_host(lay.v_new.index_select(0, tok)),
                                      W.to_host(pool.k_cache.index_select(0, idx)),
                                      W.to_host(pool.v_cache.index_select(0, idx)), bt_c,
                                      S[rows].astype(np.int32), qsl_c)
    got_k = W.to_host(run.kc.index_select(0, idx.to(run.kc.device)))
    got_v = W.to_host(run.vc.index_select(0, idx.to(run.vc.device)))
    assert np.array_equal(got_k, want_k), f"k pages differ after the append (layer {layer})"
    assert np.array_equal(got_v, want_v), f"v pages differ after the append (layer {layer})"
    return int(touched.shape[0])


def _sampled_check(batch, rows, n_per_row, seed, layer=0, run=None):
    if run is None:
        run = Run(batch, layer)
        run.append()
        run.forward()
    code, bits = run.status()
    assert code == 0, f"device status bits {bits}"
    rng = np.random.default_rng(seed)
    toks, heads, ref_out, ref_lse = oracle_sampled(batch, rows, n_per_row, rng, layer)
    got_out, got_lse = run.out_host()
    return assert_parity(got_out[toks, heads], got_lse[toks, heads], ref_out, ref_lse,
                         f"{batch.name} layer {layer}")


def test_decode_batch_full():
    b = W.config_decode(device="cuda")
    run = Run(b)
    run.append()
    run.forward()
    code, _ = run.status()
    assert code == 0
    ref_out, ref_lse, _ = oracle_full(b)
    got_out, got_lse = run.out_host()
    assert_parity(got_out, got_lse, ref_out, ref_lse, "decode_b64")


def test_mixed_batch_sampled():
    b = W.config_mixed(device="cuda")
    L = b.q_lens
    app = list(np.nonzero(L > 1)[0])
    dec = list(np.nonzero(L == 1)[0])
    rng = np.random.default_rng(5)
    rows = sorted(app[:6] + list(rng.choice(dec, size=10, replace=False)))
    run = Run(b)
    run.append()
    run.forward()
    # the whole step's KV append, every written page bit for bit
    assert _appended_pages_bitexact(b, run) > 1000
    _sampled_check(b, rows, n_per_row=24, seed=6, run=run)


def test_long_horizon_sampled():
    b = W.config_long(device="cuda")
    order = np.argsort(b.seq_lens)
    rows = sorted(list(order[:3]) + list(order[-4:]) + list(order[len(order) // 2: len(order) // 2 + 3]))
    _sampled_check(b, rows, n_per_row=16, seed=7)


def test_rollout_step_sampled_every_layer():
    b = W.config_rollout(device="cuda")
    L = b.q_lens
    rng = np.random.default_rng(8)
    app = list(np.nonzero(L > 1)[0])
    dec = list(np.nonzero(L == 1)[0])
    # one whole GRPO group (shared prompt) plus a few others
    grp_rows = list(np.nonzero(b.group_of_row == b.group_of_row[dec[0]])[0])
    rows = sorted(set(grp_rows + app[:3] + list(rng.choice(dec, size=4, replace=False))))
    for layer in range(len(b.layers)):
        run = Run(b, layer)
        run.append()
        run.forward()
        if b.layers[layer].sliding_window == 0:
            assert run.header()["n_cascade"] > 0
        _appended_pages_bitexact(b, run, layer)
        _sampled_check(b, rows, n_per_row=6, seed=100 + layer, layer=layer, run=run)
        del run
        torch.cuda.empty_cache()


# ------------------------------------------------------------ CUDA graphs


def test_cuda_graph_replay_follows_new_lengths():
    # KV append + forward captured once; the planner runs inside the graph, so
    # a replay after seq_lens changed (same dims) computes the new batch
    import dataclasses

    rng = np.random.default_rng(61)
    B = 12
    S = rng.integers(200, 3000, size=B)
    L = np.where(np.arange(B) % 3 == 0, np.minimum(S - 150, rng.integers(2, 300, size=B)), 1)
    b = W.build_batch("graph", 62, S, L, 64, 8)
    run = Run(b)
    k0, v0 = run.kc.clone(), run.vc.clone()
    run.append()
    run.forward()
    assert run.status()[0] == 0
    out_e, lse_e = run.out_host()

    run.kc.copy_(k0)
    run.vc.copy_(v0)
    torch.cuda.synchronize()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(mcpu.NUM_PHASE_EVENTS)]
    for e in ev:  # torch creates the CUDA event at its first record
        e.record()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        run.append()
        mcpu.mcpu_paged_attention_forward(run.q, run.kc, run.vc, run.bt, run.sl, run.qsl, run.window,
                                          b.softmax_scale, run.out, run.lse, run.ws, phase_events=ev)
    run.out.fill_(float("nan"))
    g.replay()
    assert run.status()[0] == 0
    out_g, lse_g = run.out_host()
    assert np.array_equal(out_g, out_e) and np.array_equal(lse_g, lse_e)
    assert ev[0].elapsed_time(ev[5]) > 0  # the phase events are graph nodes

    # shorter contexts, same chunks and pages: replay the same graph
    S2 = (S - rng.integers(1, 150, size=B)).astype(np.int32)
    b2 = dataclasses.replace(b, seq_lens=S2)
    run.kc.copy_(k0)
    run.vc.copy_(v0)
    run.sl.copy_(torch.from_numpy(S2))
    run.out.fill_(float("nan"))
    g.replay()
    assert run.status()[0] == 0
    ref_out, ref_lse, (okc, ovc) = oracle_full(b2)
    assert np.array_equal(W.to_host(run.kc), okc) and np.array_equal(W.to_host(run.vc), ovc)
    got_out, got_lse = run.out_host()
    assert_parity(got_out, got_lse, ref_out, ref_lse, "graph replay, new lengths")
    assert np.abs(got_out - out_e).max() > 0  # the replay did compute the new batch


# ------------------------------------------------------- attention sinks


def _sinks(hq, seed):
    return np.random.default_rng(seed).normal(0.0, 1.5, size=hq).astype(np.float32)


@pytest.mark.parametrize("seed", range(8))
def test_sinks_fuzz(seed):
    b = W.fuzz_batch(900 + seed, max_len=2000, max_chunk=200)
    _full_check(b, what=f"sinks fuzz{seed}", sinks=_sinks(b.num_q_heads, seed))


@pytest.mark.parametrize("split_pages", [1, 3])
def test_sinks_on_split_rows(split_pages):
    # split rows take their sink in the merge, unsplit rows in the decode kernel
    b = W.build_batch("sinksplit", 56, [700, 33, 2049, 16, 1], [1, 1, 1, 1, 1], 32, 8)
    run, _ = _full_check(b, split_pages=split_pages, what=f"sinks split{split_pages}", sinks=_sinks(32, 1))
    assert run.header()["n_merge"] > 0


def test_sinks_with_cascade_groups():
    b = _grouped_batch(4)
    run, _ = _full_check(b, what="sinks cascade", sinks=_sinks(64, 2))
    assert run.header()["n_cascade"] > 0


@pytest.mark.parametrize("window", [16, 128])
def test_sinks_with_windows(window):
    rng = np.random.default_rng(window + 5)
    S = rng.integers(1, 2500, size=6)
    L = np.where(np.arange(6) % 2 == 0, 1, np.minimum(S, rng.integers(2, 300, size=6)))
    b = W.build_batch("sinkwin", 78 + window, S, L, 64, 8, layer_windows=(window,))
    _full_check(b, what=f"sinks window{window}", sinks=_sinks(64, 3))


def test_sinks_on_both_append_kernels():
    rng = np.random.default_rng(57)
    S = rng.integers(200, 3000, size=4)
    L = np.minimum(S, rng.integers(2, 400, size=4))
    b = W.build_batch("sinkapp", 58, S, L, 16, 2)
    sk = _sinks(16, 4)
    _full_check(b, what="sinks tcgen05 append", sinks=sk)
    _full_check(b, flags=mcpu.FLAG_MMA_SYNC_APPEND, what="sinks mma.sync append", sinks=sk)


def test_sinks_mixed_batch_sampled():
    b = W.config_mixed(device="cuda")
    sk = _sinks(b.num_q_heads, 5)
    run = Run(b)
    run.append()
    run.forward(sinks=sk)
    assert run.status()[0] == 0
    L = b.q_lens
    app = list(np.nonzero(L > 1)[0])
    dec = list(np.nonzero(L == 1)[0])
    rows = sorted(app[:4] + dec[:6])
    rng = np.random.default_rng(12)
    toks, heads, ref_out, ref_lse = oracle_sampled(b, rows, 16, rng, sinks=sk)
    got_out, got_lse = run.out_host()
    assert_parity(got_out[toks, heads], got_lse[toks, heads], ref_out, ref_lse, "mixed with sinks")


# ------------------------------------------------- bad inputs and limits


def _good_rows_parity(run, b, good, what):
    rng = np.random.default_rng(77)
    toks, heads, ref_out, ref_lse = oracle_sampled(b, good, 24, rng)
    got_out, got_lse = run.out_host()
    assert_parity(got_out[toks, heads], got_lse[toks, heads], ref_out, ref_lse, what)


def test_bad_page_ids_are_reported_and_other_rows_are_unaffected():
    # pages outside the pool (too large, negative) in a decode row and in an
    # append row: the kernels check every page id, load zeros instead and
    # raise MCPU_ERR_BAD_PAGE; rows with valid tables are computed as usual
    S = [900, 300, 1200, 77, 500, 260]
    L = [1, 40, 1, 1, 90, 1]
    b = W.build_batch("badpage", 71, S, L, 16, 2)
    run = Run(b)
    n_pages = run.kc.shape[0]
    run.bt[0, 3] = n_pages + 3
    run.bt[1, 10] = -7
    run.append()
    run.forward()
    code, bits = run.status()
    assert code == 5, (code, bits)  # MCPU_ERR_BAD_PAGE
    assert bits & mcpu.STATUS_BAD_PAGE
    _good_rows_parity(run, b, [2, 3, 4, 5], "rows next to bad pages")


def test_inconsistent_lengths_are_reported():
    S = [400, 300, 700, 50]
    L = [1, 30, 1, 1]
    b = W.build_batch("badlen", 72, S, L, 16, 2)
    run = Run(b)
    run.sl[1] = 10  # L = 30 > S = 10: the row is skipped
    run.append()
    run.forward()
    code, bits = run.status()
    assert code == 6 and bits & mcpu.STATUS_BAD_LENGTHS, (code, bits)  # MCPU_ERR_BAD_LENGTHS
    _good_rows_parity(run, b, [0, 2, 3], "rows next to a bad length")
    # query_start_loc that does not end at total_q: nothing is planned
    run2 = Run(b)
    run2.qsl[-1] = int(b.total_q) - 1
    run2.forward()
    code, bits = run2.status()
    assert code == 6 and bits & mcpu.STATUS_BAD_LENGTHS
    assert run2.header()["n_decode"] == 0 and run2.header()["n_append"] == 0


def test_largest_row_count():
    # 2048 rows (the planner's limit), short decode and append rows mixed
    rng = np.random.default_rng(73)
    B = 2048
    S = rng.integers(1, 400, size=B)
    L = np.where(rng.random(B) < 0.05, np.minimum(S, rng.integers(2, 40, size=B)), 1)
    b = W.build_batch("rows2048", 74, S, L, 16, 2)
    run = Run(b)
    run.append()
    run.forward()
    assert run.status()[0] == 0
    rows = sorted(rng.choice(B, size=40, replace=False))
    _good_rows_parity(run, b, rows, "2048 rows")


@pytest.mark.parametrize("layer", [0, 1])
def test_programmatic_launches_match_ordinary_ones_bitwise(layer):
    # Without phase events the planner (after the prefix scan), the cascade
    # pass (after the decode kernel) and the merge (after the cascade pass)
    # are programmatic launches that overlap the grid before them; with phase
    # events every kernel is an ordinary launch. Layer 1 of the rollout
    # profiling batch has GRPO groups (cascade items) and split rows; layer 0
    # is a sliding-window layer. Results must agree bit for bit, eagerly and
    # as a replayed CUDA graph of the programmatic form.
    b = W.config_rollout_small(device="cpu")
    run = Run(b, layer)
    run.append()
    run.forward()
    assert run.status()[0] == 0
    if layer == 1:
        assert run.header()["n_cascade"] > 0 and run.header()["n_merge"] > 0
    out_p, lse_p = run.out_host()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(mcpu.NUM_PHASE_EVENTS)]
    for e in ev:  # torch creates the CUDA event at its first record
        e.record()
    run.out.fill_(float("nan"))
    mcpu.mcpu_paged_attention_forward(run.q, run.kc, run.vc, run.bt, run.sl, run.qsl, run.window,
                                      b.softmax_scale, run.out, run.lse, run.ws, phase_events=ev)
    torch.cuda.synchronize()
    assert run.status()[0] == 0
    out_o, lse_o = run.out_host()
    assert np.array_equal(out_p, out_o) and np.array_equal(lse_p, lse_o)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        run.forward()
    run.out.fill_(float("nan"))
    g.replay()
    torch.cuda.synchronize()
    assert run.status()[0] == 0
    out_g, lse_g = run.out_host()
    assert np.array_equal(out_p, out_g) and np.array_equal(lse_p, lse_g)


def _random_batch(seed):
    """Decode and append rows of random lengths, sometimes GRPO groups sharing
    prompt pages, sometimes a window; GQA group 8, 4, 2 or 1."""
    rng = np.random.default_rng(seed)
    groups, gs, B0 = int(rng.integers(0, 4)), int(rng.choice([2, 4, 8])), int(rng.integers(4, 24))
    S = rng.integers(1, 6000, size=B0)
    L = np.where(rng.random(B0) < 0.6, 1, np.minimum(S, rng.integers(2, 400, size=B0)))
    kw = {}
    if groups:
        prompt = np.repeat(rng.integers(40, 2500, size=groups), gs)
        Sg = prompt + rng.integers(1, 1500, size=groups * gs)
        Lg = np.minimum(np.where(rng.random(groups * gs) < 0.8, 1, rng.integers(2, 100, size=groups * gs)), Sg)
        S, L = np.concatenate([Sg, S]), np.concatenate([Lg, L])
        kw = dict(shared_prefix_pages=np.concatenate([prompt // 16, np.zeros(B0, np.int64)]),
                  prompt_lens=np.concatenate([prompt, np.zeros(B0, np.int64)]),
                  group_of_row=np.concatenate([np.repeat(np.arange(groups), gs), -np.ones(B0, np.int64)]))
    hq, hkv = [(64, 8), (32, 8), (16, 8), (8, 8)][int(rng.integers(0, 4))]
    win = int(rng.choice([0, 0, 0, 128, 1000])) if not groups else 0
    sinks = rng.normal(0, 2, size=hq).astype(np.float32) if seed % 3 == 0 else None
    return W.build_batch("random", seed, S, L, hq, hkv, layer_windows=(win,), **kw), sinks


@pytest.mark.parametrize("seed", [9001, 9003, 9005, 9007, 9008, 9014])
def test_random_batches_with_groups_windows_and_sinks(seed):
    # seeds chosen for: window 128 (g 2), groups + sinks (g 8), groups (g 8),
    # groups (g 4), window 1000 (g 8), plain (g 1); each against the oracle on
    # all outputs, the pools bit for bit, and the side-stream and
    # single-stream launch orders bit for bit against each other
    b, sinks = _random_batch(seed)
    run, _ = _full_check(b, sinks=sinks, what=f"random{seed}")
    out1, lse1 = run.out_host()
    run.forward(flags=mcpu.FLAG_SERIAL, sinks=sinks)
    assert run.status()[0] == 0
    out2, lse2 = run.out_host()
    assert np.array_equal(out1, out2) and np.array_equal(lse1, lse2)
