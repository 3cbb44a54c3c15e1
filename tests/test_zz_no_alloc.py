"""The forward entry point that allocates nothing, against the regular one.

mcpu_paged_attention_forward_noalloc serves callers that cannot allocate
device memory (an engine that has reserved all GPU memory, code running under
stream capture): it keeps its scratch in the library's own fixed device array
instead of a caller workspace. These tests call it through the C ABI twice in
a row, on different batches (the array keeps the previous call's contents),
and check each result against the CPU oracle and against
mcpu_paged_attention_forward at the tolerances of the other parity tests;
decode rows as long as the long-horizon batch's (never split here) and a
batch at the token limit of the fixed scratch are covered too. This file is
collected last on purpose.
"""
import numpy as np
import pytest
import torch

import workloads as W

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    from _gpu import LSE_ABS, OUT_ABS, OUT_REL, Run, assert_parity, oracle_full, oracle_sampled
    from paper_2608_22167_gb300 import mcpu


def _noalloc(run):
    out = torch.full_like(run.q, float("nan"))
    lse = torch.full(run.q.shape[:2], float("nan"), dtype=torch.float32, device=run.q.device)
    status = torch.full((1,), -1, dtype=torch.int32, device=run.q.device)
    mcpu.mcpu_paged_attention_forward_noalloc(run.q, run.kc, run.vc, run.bt, run.sl, run.qsl, run.window,
                                              run.batch.softmax_scale, out, lse, status_word=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0, f"device status bits {int(status.item())}"
    return out.float().cpu().numpy(), lse.cpu().numpy()


def _compare(run, with_oracle=True):
    run.append()
    run.forward()
    code, bits = run.status()
    assert code == 0, bits
    ref_out, ref_lse = run.out_host()
    got_out, got_lse = _noalloc(run)
    if with_oracle:  # directly against the oracle, not only through the other entry point
        o_out, o_lse, _ = oracle_full(run.batch, run.layer)
        assert_parity(got_out, got_lse, o_out, o_lse, f"noalloc {run.batch.name} vs oracle")
    assert np.all(np.isfinite(got_out))
    err = np.abs(got_out - ref_out)
    assert err.max() <= OUT_ABS
    assert err.max() / max(np.abs(ref_out).max(), 1e-30) <= OUT_REL
    fin = np.isfinite(ref_lse)
    assert np.array_equal(fin, np.isfinite(got_lse))
    assert np.abs(got_lse[fin] - ref_lse[fin]).max() <= LSE_ABS
    return got_out, got_lse


def _grouped_batch(seed):
    rng = np.random.default_rng(seed)
    grp = np.repeat(np.arange(3), 8)
    prompt = rng.integers(100, 1200, size=3)[grp]
    L = np.where(rng.random(24) < 0.25, rng.integers(2, 100, size=24), 1)
    S = prompt + rng.integers(0, 600, size=24) + L
    return W.build_batch("noalloc_groups", seed, S, L, 64, 8, shared_prefix_pages=prompt // 16, prompt_lens=prompt,
                         group_of_row=grp)


def test_two_calls_in_a_row_match_the_workspace_entry_point():
    # call 1: a mixed batch (long decode rows, append chunks) of 64q/8kv heads
    rng = np.random.default_rng(11)
    S = rng.integers(1, 6000, size=9)
    L = np.where(np.arange(9) % 3 == 0, np.minimum(S, rng.integers(2, 400, size=9)), 1)
    first = Run(W.build_batch("noalloc_mixed", 12, S, L, 64, 8))
    out1, lse1 = _compare(first)
    # call 2: a different batch (GRPO groups sharing prompt pages; the regular
    # entry point runs its cascade pass here, this one does not)
    second = Run(_grouped_batch(13))
    _compare(second)
    # and the first batch once more: same bits as its first call
    out1b, lse1b = _noalloc(first)
    assert np.array_equal(out1, out1b) and np.array_equal(lse1, lse1b)


@pytest.mark.parametrize("window", [0, 128])
def test_window_and_small_heads(window):
    b = W.build_batch("noalloc_small", 21 + window, [17, 300, 129, 64], [1, 30, 1, 64], 8, 2,
                      layer_windows=(window,))
    run = Run(b)
    _compare(run)
    _compare(run)


def test_long_decode_rows_are_served_unsplit():
    # decode rows of 49152-65536 keys (the long-horizon batch's longest),
    # each read by one warp per kv head here: within tolerance of the oracle
    # and of the split workspace path, and no wait runs out
    S = [65536, 49153, 3000, 700]
    L = [1, 1, 200, 1]
    run = Run(W.build_batch("noalloc_long", 31, S, L, 64, 8, device="cuda"))
    _compare(run)


def test_token_limit_of_the_fixed_scratch():
    # total_q exactly at the limit (262144 query tokens: four 65536-token
    # append chunks): the plan fits the fixed scratch and the results equal
    # the workspace path's bit for bit (same kernels, no decode rows)
    S = [65536] * 4
    b = W.build_batch("noalloc_limit", 32, S, S, 64, 8, device="cuda")
    assert b.total_q == 262144
    run = Run(b)
    run.append()
    run.forward()
    assert run.status()[0] == 0
    out = torch.full_like(run.q, float("nan"))
    lse = torch.full(run.q.shape[:2], float("nan"), dtype=torch.float32, device=run.q.device)
    status = torch.full((1,), -1, dtype=torch.int32, device=run.q.device)
    mcpu.mcpu_paged_attention_forward_noalloc(run.q, run.kc, run.vc, run.bt, run.sl, run.qsl, 0, b.softmax_scale,
                                              out, lse, status_word=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    # compared on the device (2 GiB of outputs)
    assert torch.equal(out.view(torch.int16), run.out.view(torch.int16))
    assert torch.equal(lse.view(torch.int32), run.lse.view(torch.int32))
    rng = np.random.default_rng(33)
    toks, heads, o_out, o_lse = oracle_sampled(b, [0, 3], 12, rng)
    t_ = torch.as_tensor(toks, device=out.device)
    h_ = torch.as_tensor(heads.astype(np.int64), device=out.device)
    assert_parity(out[t_, h_].float().cpu().numpy(), lse[t_, h_].cpu().numpy(), o_out, o_lse,
                  "noalloc at the token limit, sampled")


def test_rejects_what_does_not_fit():
    b = W.config_tiny()
    run = Run(b)
    d = mcpu.dims(run.q, run.kc, run.bt, run.sl)
    d.total_q = 262145  # beyond the fixed scratch's limit: rejected before any launch
    import ctypes
    code = mcpu._lib.mcpu_paged_attention_forward_noalloc(
        mcpu._ptr(run.q), mcpu._ptr(run.kc), mcpu._ptr(run.vc), mcpu._ptr(run.bt), mcpu._ptr(run.sl),
        mcpu._ptr(run.qsl), 0, 0.125, ctypes.byref(d), mcpu._ptr(run.out), mcpu._ptr(run.lse), None,
        mcpu._stream(None))
    assert code == 3  # MCPU_ERR_WORKSPACE_TOO_SMALL
