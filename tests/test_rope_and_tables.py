"""Fused RoPE + KV append and device-side block-table growth on the GPU,
against the oracle's rotation and a plain model of the page stack."""
import numpy as np
import pytest
import torch

import workloads as W

pytestmark = pytest.mark.gpu

if torch.cuda.is_available():
    import oracle
    from _gpu import Run, assert_parity
    from paper_2608_22167_gb300 import mcpu


def _bits(t):
    return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def _f(bits):
    return oracle.bf16_bits_to_float(bits).astype(np.float64)


def _pair_magnitude(x_bits):
    x = np.abs(_f(x_bits))
    m = x[..., :32] + x[..., 32:]
    return np.concatenate([m, m], axis=-1)


def _assert_rotation_close(got_bits, ref_bits, in_bits, ref_in=None):
    g, r = _f(got_bits), _f(ref_bits)
    mag = _pair_magnitude(in_bits) if in_bits is not None else ref_in
    assert np.all(np.abs(g - r) <= 2.0**-7 * np.abs(r) + 2.0**-21 * mag)  # one bf16 ulp + fp32 error


def _rotated_cache_inputs(h, kc_ref):
    """|x_i| + |x_{i+32}| of the unrotated input of every cache row: rows the
    append did not touch keep their values (bound from the rotated ones,
    which have the same pair magnitude up to rounding)."""
    return _pair_magnitude(kc_ref) * 1.5


@pytest.mark.parametrize("seed", range(4))
def test_rope_kv_append_matches_the_oracle(seed):
    rng = np.random.default_rng(500 + seed)
    B = 6
    S = rng.integers(2, 1500, size=B)
    L = np.where(np.arange(B) % 2 == 0, 1, np.minimum(S, rng.integers(2, 200, size=B)))
    b = W.build_batch("rope", 510 + seed, S, L, 16, 2)
    run = Run(b)
    tab = W.rope_table(int(S.max()) + 1)
    h = W.host_inputs(b)
    q = run.q.clone()
    mcpu.mcpu_rope_kv_append(q, run.k_new, run.v_new, run.kc, run.vc, run.bt, run.sl, run.qsl,
                             torch.from_numpy(tab).cuda(), mcpu.status_word(run.ws))
    assert run.status()[0] == 0
    pos = oracle.token_positions(h["seq_lens"], h["query_start_loc"])
    q_ref = oracle.rope(h["q"], pos, tab)
    k_rot = oracle.rope(h["k_new"], pos, tab)
    kc_ref, vc_ref = oracle.kv_append(k_rot, h["v_new"], h["k_cache"], h["v_cache"], h["block_table"],
                                      h["seq_lens"], h["query_start_loc"])
    # fp32 on the GPU, fp64 in the oracle, each rounded once to bf16: apart by
    # at most one rounding of the result plus the fp32 error of a c - b s
    _assert_rotation_close(_bits(q), q_ref, h["q"])
    _assert_rotation_close(_bits(run.kc), kc_ref, None, ref_in=_rotated_cache_inputs(h, kc_ref))
    assert np.array_equal(_bits(run.vc), vc_ref)
    # attention over the rotated inputs
    run.q.copy_(q)
    run.forward()
    assert run.status()[0] == 0
    ref_out, ref_lse = oracle.paged_attention(q_ref, kc_ref, vc_ref, h["block_table"], h["seq_lens"],
                                              h["query_start_loc"], 0, b.softmax_scale)
    got_out, got_lse = run.out_host()
    assert_parity(got_out, got_lse, oracle.bf16_bits_to_float(ref_out), ref_lse, "after rope append")


def test_rope_positions_past_the_table_are_reported():
    b = W.build_batch("ropebad", 520, [40, 300], [1, 20], 16, 2)
    run = Run(b)
    tab = torch.from_numpy(W.rope_table(100)).cuda()  # row 1 reaches position 299
    q = run.q.clone()
    mcpu.mcpu_rope_kv_append(q, run.k_new, run.v_new, run.kc, run.vc, run.bt, run.sl, run.qsl, tab,
                             mcpu.status_word(run.ws))
    code, bits = run.status()
    assert code == 6 and bits & mcpu.STATUS_BAD_LENGTHS
    assert torch.equal(q[1:], run.q[1:])  # row 1's tokens are left alone


def _grow_case(seed, n_free):
    rng = np.random.default_rng(seed)
    B, maxp = 40, 64
    S = rng.integers(0, maxp * 16, size=B).astype(np.int32)
    bt = np.full((B, maxp), -1, np.int32)
    used = rng.permutation(100000)
    k = 0
    for r in range(B):  # some leading pages already in place, the first 4 rows share theirs
        have = int(rng.integers(0, (S[r] + 15) // 16 + 1))
        for j in range(have):
            bt[r, j] = used[j] if r < 4 else used[1000 + k]
            k += 0 if r < 4 else 1
    free = used[50000:50000 + n_free].astype(np.int32)
    return S, bt, free


@pytest.mark.parametrize("n_free", [4000, 60])
def test_grow_block_tables(n_free):
    S, bt, free = _grow_case(9, n_free)
    dev = torch.device("cuda")
    bt_d = torch.from_numpy(bt).to(dev)
    count = torch.tensor([len(free)], dtype=torch.int32, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    mcpu.mcpu_grow_block_tables(bt_d, torch.from_numpy(S).to(dev), torch.from_numpy(free).to(dev), count, status)
    got = bt_d.cpu().numpy()
    need = (S.astype(np.int64) + 15) // 16
    missing = sum(int((bt[r, :need[r]] < 0).sum()) for r in range(len(S)))
    left = int(count.item())
    n_new = len(free) - left
    assert n_new == min(missing, len(free))
    for r in range(len(S)):
        pre = bt[r] >= 0
        assert np.array_equal(got[r][pre], bt[r][pre])          # entries already set are untouched
        assert np.all(got[r, need[r]:] == -1)                   # nothing past the row's length
    new = got[(bt < 0) & (got >= 0)]
    assert sorted(new.tolist()) == sorted(free[left:].tolist())  # exactly the top of the stack, each once
    if missing > len(free):
        assert int(status.item()) & mcpu.STATUS_POOL_EXHAUSTED and left == 0
    else:
        assert int(status.item()) == 0
        assert all(np.all(got[r, :need[r]] >= 0) for r in range(len(S)))
