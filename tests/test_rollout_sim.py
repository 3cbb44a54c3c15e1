"""The rollout simulator's bookkeeping on the CPU, and the CUDA path driven
by it for many steps of a continuously changing batch on the GPU."""
import collections

import numpy as np
import pytest
import torch

from paper_2608_22167_gb300.rollout_sim import PAGE, RolloutSim, SimConfig


def _small_cfg(**kw):
    base = dict(num_pages=4096, max_pages_per_seq=256, max_live_groups=3, group_size=4, prompt_len=(40, 400),
                response_len=(2, 12), observation_len=(20, 120), tool_wait_steps=(1, 4), acquire_steps=(0, 2),
                max_turns=(1, 3), max_len=2000)
    base.update(kw)
    return SimConfig(**base)


def _check_pages(sim):
    refs = collections.Counter()
    for t in sim.trajs.values():
        assert len(set(t.pages)) == len(t.pages), "a page twice in one block table"
        refs.update(t.pages)
    for p, n in refs.items():
        assert sim.pool.refs[p] == n
    assert int(sim.pool.refs.sum()) == sum(refs.values())
    free = set(sim.pool.free)
    assert not free & set(refs)
    assert len(free) + len(refs) == sim.cfg.num_pages


def test_bookkeeping_over_many_steps():
    sim = RolloutSim(_small_cfg(), seed=3)
    length = {}
    kinds = collections.Counter()
    for _ in range(300):
        b = sim.step()
        _check_pages(sim)
        assert np.all(b.q_lens >= 1) and np.all(b.q_lens <= b.seq_lens)
        # groups are contiguous in the batch
        seen, prev = set(), None
        for g in b.groups:
            if g != prev:
                assert g not in seen
                seen.add(g)
                prev = g
        for i, tid in enumerate(b.tids):
            S, L = int(b.seq_lens[i]), int(b.q_lens[i])
            n_pages = (S + PAGE - 1) // PAGE
            assert np.all(b.block_table[i, :n_pages] >= 0) and np.all(b.block_table[i, n_pages:] == -1)
            if tid in length:
                assert S == length[tid] + L, "a row grows by exactly its query tokens"
            length[int(tid)] = S
            kinds["decode" if L == 1 else "append"] += 1
    assert sim.finished > 0 and kinds["decode"] > 0 and kinds["append"] > 0


def test_group_members_share_full_prompt_pages():
    sim = RolloutSim(_small_cfg(prompt_len=(200, 200), acquire_steps=(0, 0)), seed=5)
    b = sim.step()  # every group's prefill step
    for g in np.unique(b.groups):
        rows = np.nonzero(b.groups == g)[0]
        assert len(rows) == sim.cfg.group_size  # 200 % 16 != 0: every member appends its tail
        full = 200 // PAGE
        for r in rows[1:]:
            assert np.array_equal(b.block_table[r, :full], b.block_table[rows[0], :full])
            assert b.block_table[r, full] != b.block_table[rows[0], full]  # private tail page
        assert b.q_lens[rows[0]] == 200 and np.all(b.q_lens[rows[1:]] == 200 - full * PAGE)


def test_pool_drains_to_empty():
    sim = RolloutSim(_small_cfg(), seed=8)
    for _ in range(40):
        sim.step()
    sim.cfg.max_live_groups = 0  # admit nothing more
    for _ in range(2000):
        if not sim.trajs:
            break
        sim.step()
    assert not sim.trajs and sim.pool.in_use == 0


# ------------------------------------------------------------------ GPU


@pytest.mark.gpu
def test_cuda_path_under_churn_matches_the_oracle():
    import oracle
    from _gpu import assert_parity
    from paper_2608_22167_gb300 import mcpu

    dev = torch.device("cuda")
    cfg = _small_cfg(num_pages=4096, max_live_groups=4, group_size=8, prompt_len=(100, 900))
    sim = RolloutSim(cfg, seed=11)
    Hq, Hkv, D = 64, 8, 64
    gen = torch.Generator(device=dev)
    gen.manual_seed(12)
    kc = torch.randn((cfg.num_pages, Hkv, PAGE, D), generator=gen, device=dev, dtype=torch.bfloat16)
    vc = torch.randn((cfg.num_pages, Hkv, PAGE, D), generator=gen, device=dev, dtype=torch.bfloat16)
    rng = np.random.default_rng(13)
    checks = 0
    for step in range(36):
        b = sim.step()
        if b.num_seqs == 0:
            continue
        T = b.total_q
        q = torch.randn((T, Hq, D), generator=gen, device=dev, dtype=torch.bfloat16)
        kn = torch.randn((T, Hkv, D), generator=gen, device=dev, dtype=torch.bfloat16)
        vn = torch.randn((T, Hkv, D), generator=gen, device=dev, dtype=torch.bfloat16)
        bt = torch.from_numpy(b.block_table).to(dev)
        sl = torch.from_numpy(b.seq_lens).to(dev)
        qsl = torch.from_numpy(b.query_start_loc).to(dev)
        d = mcpu.dims(q, kc, bt, sl)
        ws = mcpu.new_workspace(d, dev)
        out = torch.empty_like(q)
        lse = torch.empty((T, Hq), dtype=torch.float32, device=dev)
        check = step % 6 == 5
        if check:
            k_before = kc.view(torch.int16).cpu().numpy().view(np.uint16)
            v_before = vc.view(torch.int16).cpu().numpy().view(np.uint16)
        mcpu.mcpu_kv_append(kn, vn, kc, vc, bt, sl, qsl, mcpu.status_word(ws))
        mcpu.mcpu_paged_attention_forward(q, kc, vc, bt, sl, qsl, 0, 0.125, out, lse, ws)
        code, bits = mcpu.mcpu_read_device_status(ws)
        assert code == 0, f"step {step}: device status {bits}"
        if not check:
            continue
        checks += 1
        host = lambda t: t.view(torch.int16).cpu().numpy().view(np.uint16)  # noqa: E731
        okc, ovc = oracle.kv_append(host(kn), host(vn), k_before, v_before, b.block_table, b.seq_lens,
                                    b.query_start_loc)
        assert np.array_equal(host(kc), okc) and np.array_equal(host(vc), ovc), f"step {step}: KV append"
        n = 256
        toks = rng.integers(0, T, size=n).astype(np.int64)
        heads = rng.integers(0, Hq, size=n).astype(np.int32)
        ro, rl = oracle.paged_attention_sampled(host(q), okc, ovc, b.block_table, b.seq_lens, b.query_start_loc,
                                                0, 0.125, toks, heads)
        go = out.float().cpu().numpy()[toks, heads]
        gl = lse.cpu().numpy()[toks, heads]
        assert_parity(go, gl, oracle.bf16_bits_to_float(ro), rl, f"churn step {step}")
    assert checks >= 5
