"""GPU: mcpu_paged_attention_host (per-token inputs and outputs in host
memory, copies overlapped with the compute by row slices) against the CPU
oracle on the same seeded inputs: outputs within the tolerances, KV pools
bit for bit, several calls in flight on one stage, and its argument checks."""
import numpy as np
import pytest
import torch

import workloads as W

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    from _gpu import assert_parity, oracle_full, oracle_sampled
    from paper_2608_22167_gb300 import mcpu


class HostCall:
    """One layer of a batch as host tensors (page-locked) plus device pools."""

    def __init__(self, batch, layer=0, pinned=True):
        lay = batch.layers[layer]
        pool = batch.pools[lay.pool]
        pin = (lambda t: t.pin_memory()) if pinned else (lambda t: t)
        self.batch, self.layer = batch, layer
        self.q = pin(lay.q.cpu().contiguous())
        self.k_new = pin(lay.k_new.cpu().contiguous())
        self.v_new = pin(lay.v_new.cpu().contiguous())
        self.kc = pool.k_cache.to("cuda").clone()
        self.vc = pool.v_cache.to("cuda").clone()
        self.bt = torch.from_numpy(pool.block_table).to("cuda")
        self.sl = torch.from_numpy(batch.seq_lens).to(torch.int32)
        self.qsl = torch.from_numpy(batch.query_start_loc).to(torch.int32)
        self.window = lay.sliding_window
        self.out = pin(torch.full(self.q.shape, float("nan"), dtype=torch.bfloat16))
        self.lse = pin(torch.full(self.q.shape[:2], float("nan"), dtype=torch.float32))
        self.dims = mcpu.dims(self.q, self.kc, self.bt, self.sl)
        self.ws = mcpu.new_workspace(self.dims, "cuda")

    def stage(self):
        return mcpu.HostStage(max(1, self.q.shape[0]), max(1, self.sl.shape[0]), self.q.shape[1], self.kc.shape[1])

    def call(self, stage, slices=0):
        mcpu.mcpu_paged_attention_host(stage, self.q, self.k_new, self.v_new, self.kc, self.vc, self.bt, self.sl,
                                       self.qsl, self.window, self.batch.softmax_scale, self.out, self.lse, self.ws,
                                       slices=slices)

    def check(self, what):
        code, bits = mcpu.mcpu_read_device_status(self.ws)
        assert code == 0, f"{what}: device status bits {bits}"
        ref_out, ref_lse, (okc, ovc) = oracle_full(self.batch, self.layer)
        assert np.array_equal(W.to_host(self.kc), okc), f"{what}: k pool differs after append"
        assert np.array_equal(W.to_host(self.vc), ovc), f"{what}: v pool differs after append"
        return assert_parity(self.out.float().numpy(), self.lse.numpy(), ref_out, ref_lse, what)


@pytest.mark.parametrize("slices", [1, 2, 3, 8])
@pytest.mark.parametrize("seed", range(6))
def test_host_call_matches_oracle(seed, slices):
    b = W.fuzz_batch(3000 + seed, max_len=1200, max_chunk=200)
    hc = HostCall(b)
    st = hc.stage()
    hc.call(st, slices=slices)
    mcpu.mcpu_host_stage_sync(st)
    hc.check(f"fuzz{seed} slices={slices}")
    st.close()


@pytest.mark.parametrize("window", [0, 16, 128])
def test_host_call_with_sinks_and_windows(window):
    # options reach every slice: attention sinks, and a sliding window
    rng = np.random.default_rng(3600 + window)
    S = rng.integers(20, 1500, size=7)
    L = np.where(rng.random(7) < 0.5, 1, np.minimum(S, rng.integers(2, 200, size=7)))
    b = W.build_batch("host_sinks", 3600 + window, S, L, 16, 2, layer_windows=(window,))
    sinks = rng.normal(0.0, 2.0, size=16).astype(np.float32)
    hc = HostCall(b)
    st = hc.stage()
    mcpu.mcpu_paged_attention_host(st, hc.q, hc.k_new, hc.v_new, hc.kc, hc.vc, hc.bt, hc.sl, hc.qsl, hc.window,
                                   b.softmax_scale, hc.out, hc.lse, hc.ws, slices=3,
                                   sinks=torch.from_numpy(sinks).to("cuda"))
    mcpu.mcpu_host_stage_sync(st)
    code, bits = mcpu.mcpu_read_device_status(hc.ws)
    assert code == 0, f"device status bits {bits}"
    ref_out, ref_lse, _ = oracle_full(b, 0, sinks=sinks)
    assert_parity(hc.out.float().numpy(), hc.lse.numpy(), ref_out, ref_lse, f"sinks window={window}")
    st.close()


def test_host_call_pageable_buffers():
    # page-locked memory is the fast path, ordinary host memory must work too
    b = W.fuzz_batch(3100, max_len=800, max_chunk=100)
    hc = HostCall(b, pinned=False)
    st = hc.stage()
    hc.call(st, slices=2)
    mcpu.mcpu_host_stage_sync(st)
    hc.check("pageable")
    st.close()


@pytest.mark.parametrize("pinned", [True, False])
def test_direct_outputs_equal_the_staged_ones_bitwise(pinned):
    # MCPU_FLAG_HOST_OUT_DIRECT: the kernels write out / lse straight into
    # page-locked host memory (ordinary host memory falls back to the copies);
    # the same kernels run either way, so the results are identical
    b = W.fuzz_batch(3300 + int(pinned), max_len=1500, max_chunk=300)
    hc = HostCall(b, pinned=pinned)
    st = hc.stage()
    hc.call(st, slices=2)
    mcpu.mcpu_host_stage_sync(st)
    hc.check("staged outputs")
    ref_out, ref_lse = hc.out.clone(), hc.lse.clone()
    hc.out.fill_(float("nan"))
    hc.lse.fill_(float("nan"))
    hc.kc.copy_(b.pools[b.layers[0].pool].k_cache.to("cuda"))
    hc.vc.copy_(b.pools[b.layers[0].pool].v_cache.to("cuda"))
    mcpu.mcpu_reset_device_status(hc.ws)
    mcpu.mcpu_paged_attention_host(st, hc.q, hc.k_new, hc.v_new, hc.kc, hc.vc, hc.bt, hc.sl, hc.qsl, hc.window,
                                   b.softmax_scale, hc.out, hc.lse, hc.ws, flags=mcpu.FLAG_HOST_OUT_DIRECT)
    mcpu.mcpu_host_stage_sync(st)
    hc.check("direct outputs")
    assert torch.equal(hc.out.view(torch.int16), ref_out.view(torch.int16))
    assert torch.equal(hc.lse, ref_lse)
    st.close()


@pytest.mark.parametrize("window", [0, 100])
@pytest.mark.parametrize("hq,hkv", [(64, 8), (32, 8), (16, 8), (8, 8)])
def test_forward_into_host_memory_equals_device_outputs_bitwise(hq, hkv, window):
    # MCPU_FLAG_HOST_OUT_DIRECT on a forward call: out and lse are page-locked
    # host memory, and the append kernel writes each row as four 32-byte
    # stores (eight 16-byte ones when out is only 16-byte aligned, the second
    # buffer here): g = 8, 4, 2, 1 and partial last tiles. The values are
    # those of the device-output form, bit for bit.
    seq = np.array([900, 40, 2500, 16, 700, 333, 77])
    ql = np.array([1, 17, 300, 1, 45, 333, 5])
    b = W.build_batch("host_out", 3400 + hq + window, seq, ql, hq, hkv, layer_windows=(window,))
    lay = b.layers[0]
    pool = b.pools[lay.pool]
    kc, vc = pool.k_cache.to("cuda").clone(), pool.v_cache.to("cuda").clone()
    bt = torch.from_numpy(pool.block_table).to("cuda")
    sl = torch.from_numpy(b.seq_lens).to(torch.int32).to("cuda")
    qsl = torch.from_numpy(b.query_start_loc).to(torch.int32).to("cuda")
    q, kn, vn = lay.q.to("cuda"), lay.k_new.to("cuda"), lay.v_new.to("cuda")
    d = mcpu.dims(q, kc, bt, sl)
    ws = mcpu.new_workspace(d, "cuda")
    mcpu.mcpu_kv_append(kn, vn, kc, vc, bt, sl, qsl, mcpu.status_word(ws))
    out_d = torch.full_like(q, float("nan"))
    lse_d = torch.full(q.shape[:2], float("nan"), dtype=torch.float32, device="cuda")
    mcpu.mcpu_paged_attention_forward(q, kc, vc, bt, sl, qsl, window, b.softmax_scale, out_d, lse_d, ws)
    n = q.numel()
    big = torch.full((n + 16,), float("nan"), dtype=torch.bfloat16).pin_memory()
    assert big.data_ptr() % 32 == 0
    for off in (0, 8):  # 32-byte aligned, then 16 bytes past it
        out_h = big[off:off + n].view(q.shape)
        out_h.fill_(float("nan"))
        lse_h = torch.full(q.shape[:2], float("nan"), dtype=torch.float32).pin_memory()
        mcpu.mcpu_paged_attention_forward(q, kc, vc, bt, sl, qsl, window, b.softmax_scale, out_h, lse_h, ws,
                                          flags=mcpu.FLAG_HOST_OUT_DIRECT)
        torch.cuda.synchronize()
        code, bits = mcpu.mcpu_read_device_status(ws)
        assert code == 0, bits
        assert torch.equal(out_h.view(torch.int16), out_d.cpu().view(torch.int16)), off
        assert torch.equal(lse_h, lse_d.cpu()), off
    if hq == 64:  # the device-output form is checked against the oracle elsewhere for every g
        ref_out, ref_lse = oracle_full(b, 0)[:2]
        assert_parity(out_h.float().numpy(), lse_h.numpy(), ref_out, ref_lse, f"host outputs W={window}")


def test_one_slice_equals_the_device_call_bitwise():
    b = W.build_batch("host_vs_dev", 3200, np.array([900, 40, 2500, 16, 700]), np.array([1, 17, 300, 1, 1]), 64, 8)
    hc = HostCall(b)
    st = hc.stage()
    hc.call(st, slices=1)
    mcpu.mcpu_host_stage_sync(st)
    # the same kernels on device copies of the same inputs
    lay = b.layers[0]
    pool = b.pools[lay.pool]
    kc, vc = pool.k_cache.to("cuda").clone(), pool.v_cache.to("cuda").clone()
    q, kn, vn = lay.q.to("cuda"), lay.k_new.to("cuda"), lay.v_new.to("cuda")
    sl, qsl = hc.sl.to("cuda"), hc.qsl.to("cuda")
    out = torch.empty_like(q)
    lse = torch.empty(q.shape[:2], dtype=torch.float32, device="cuda")
    ws = mcpu.new_workspace(hc.dims, "cuda")
    mcpu.mcpu_kv_append(kn, vn, kc, vc, hc.bt, sl, qsl, mcpu.status_word(ws))
    mcpu.mcpu_paged_attention_forward(q, kc, vc, hc.bt, sl, qsl, lay.sliding_window, b.softmax_scale, out, lse, ws)
    torch.cuda.synchronize()
    assert torch.equal(out.cpu().view(torch.int16), hc.out.view(torch.int16))
    assert torch.equal(lse.cpu(), hc.lse)
    assert torch.equal(kc, hc.kc) and torch.equal(vc, hc.vc)
    st.close()


@pytest.mark.parametrize("slots", [2, 3, 4])
def test_calls_in_flight_take_slots_in_turn(slots):
    # five layers back to back on one stage before one sync: once every slot
    # is taken, a call's copies wait for the outputs of the call slots back
    b = W.build_batch("host_layers", 3300, np.array([1500, 300, 64, 2200, 900, 17]),
                      np.array([1, 120, 64, 1, 250, 1]), 16, 2, layer_windows=(0, 128, 0, 16, 0))
    calls = [HostCall(b, layer) for layer in range(5)]
    st = mcpu.HostStage(int(b.q_lens.sum()), b.num_seqs, 16, 2, slots=slots)
    for hc in calls:
        hc.call(st, slices=3)
    mcpu.mcpu_host_stage_sync(st)
    for i, hc in enumerate(calls):
        hc.check(f"layer {i}")
    st.close()


def test_stage_wait_orders_the_stream():
    b = W.fuzz_batch(3400, max_len=900, max_chunk=150)
    hc = HostCall(b)
    st = hc.stage()
    hc.call(st, slices=2)
    mcpu.mcpu_host_stage_wait(st)  # the current stream now waits for the output copies
    torch.cuda.current_stream().synchronize()
    hc.check("stream wait")
    st.close()


def test_mixed_batch_sampled_auto_slices():
    # the bench's mixed batch (256 rows, 32 appending) in the bench's call: auto slices
    b = W.config_mixed(device="cuda")
    hc = HostCall(b)
    st = hc.stage()
    hc.call(st)
    mcpu.mcpu_host_stage_sync(st)
    code, bits = mcpu.mcpu_read_device_status(hc.ws)
    assert code == 0, f"device status bits {bits}"
    L = b.q_lens
    rng = np.random.default_rng(9)
    app = list(np.nonzero(L > 1)[0])
    dec = list(np.nonzero(L == 1)[0])
    rows = sorted(app[:5] + list(rng.choice(dec, size=8, replace=False)))
    toks, heads, ref_out, ref_lse = oracle_sampled(b, rows, 16, rng)
    got_out = hc.out.float().numpy()[toks, heads]
    got_lse = hc.lse.numpy()[toks, heads]
    assert_parity(got_out, got_lse, ref_out, ref_lse, "mixed host call")
    st.close()


def test_host_call_argument_checks():
    b = W.fuzz_batch(3500)
    hc = HostCall(b)
    small = mcpu.HostStage(max(1, hc.q.shape[0] - 1), hc.sl.shape[0], hc.q.shape[1], hc.kc.shape[1])
    with pytest.raises(mcpu.McpuError) as e:
        hc.call(small)
    assert e.value.code == 1  # more tokens than the stage holds
    small.close()
    other = mcpu.HostStage(hc.q.shape[0], hc.sl.shape[0], hc.q.shape[1] * 2, hc.kc.shape[1])
    with pytest.raises(mcpu.McpuError) as e:
        hc.call(other)
    assert e.value.code == 1  # head counts differ from the stage's
    other.close()
    st = hc.stage()
    if hc.qsl.shape[0] > 2:
        bad = hc.qsl.clone()
        bad[1] = bad[2] + 1  # decreasing
        with pytest.raises(mcpu.McpuError) as e:
            mcpu.mcpu_paged_attention_host(st, hc.q, hc.k_new, hc.v_new, hc.kc, hc.vc, hc.bt, hc.sl, bad, 0, 0.125,
                                           hc.out, hc.lse, hc.ws)
        assert e.value.code == 1
    with pytest.raises(mcpu.McpuError) as e:
        hc.call(st, slices=mcpu.MAX_HOST_SLICES + 1)
    assert e.value.code == 1
    mcpu.mcpu_host_stage_sync(st)  # nothing enqueued: returns at once
    st.close()
