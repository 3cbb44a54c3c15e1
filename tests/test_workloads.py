"""The seeded input recipes (host only): the synthetic batches that stand in
for the paper's rollouts have the shapes and structure the recipes state.
Lengths are drawn without allocating the large pools."""
import numpy as np
import pytest

import workloads as W


@pytest.mark.parametrize("groups", [8, 48])
def test_rollout_lengths_follow_the_grpo_recipe(groups):
    S, L, grp, prompt, shared = W.rollout_lengths(groups=groups)
    B = groups * 8
    assert S.shape == L.shape == grp.shape == prompt.shape == shared.shape == (B,)
    # the 8 samples of a task are adjacent rows and share one prompt length
    assert np.array_equal(grp, np.repeat(np.arange(groups), 8))
    for g in range(groups):
        assert len(set(prompt[grp == g].tolist())) == 1
    assert prompt.min() >= 1024 and prompt.max() <= 8192
    # only full prompt pages are shared
    assert np.array_equal(shared, prompt // W.PAGE)
    # 15 % of rows append a chunk in [64, 1024]; the rest decode one token
    app = L > 1
    assert int(app.sum()) == int(round(0.15 * B))
    assert L[app].min() >= 64 and L[app].max() <= 1024
    assert np.all(L[~app] == 1)
    cont = S - prompt - L
    assert cont.min() >= 0 and cont.max() <= 24576
    # the appending rows are a seeded choice, not the first rows
    assert not np.array_equal(np.flatnonzero(app), np.arange(int(app.sum())))
    S2, L2, *_ = W.rollout_lengths(groups=groups)
    assert np.array_equal(S, S2) and np.array_equal(L, L2)


def test_tiny_config_shapes_and_page_permutation():
    b = W.config_tiny()
    assert b.num_seqs == 4 and b.total_q == 4
    assert b.seq_lens.tolist() == [17, 64, 129, 300]
    assert (b.num_q_heads, b.num_kv_heads, b.head_dim, b.page_size) == (8, 2, 64, 16)
    assert b.softmax_scale == pytest.approx(1 / 8)
    (pool,) = b.pools.values()
    assert tuple(pool.k_cache.shape[1:]) == (2, 16, 64)
    # every page a row can see is its own physical page: no page is used twice
    used = np.concatenate([pool.block_table[r, : -(-int(s) // 16)] for r, s in enumerate(b.seq_lens)])
    assert used.min() >= 0 and used.max() < pool.num_pages
    assert len(np.unique(used)) == len(used)
    # scattered, not the identity layout
    assert not np.array_equal(used, np.arange(len(used)))
    lay = b.layers[0]
    assert tuple(lay.q.shape) == (4, 8, 64) and tuple(lay.k_new.shape) == (4, 2, 64)


def test_rollout_small_draws_the_rollout_recipe_at_eight_groups():
    S, L, grp, prompt, _ = W.rollout_lengths(seed=1015, groups=8)
    assert len(S) == 64 and int((L > 1).sum()) == 10
    assert "rollout_small" in W.CONFIGS
