"""Seeded synthetic inputs for the paged-attention hot path.

This module is the only code that the CUDA path and the CPU oracle share. It
holds none of the attention arithmetic: it draws sequence lengths, allocates
physical KV pages and builds block tables (logical page -> physical page), and
fills Q, K and V with N(0, 1) bf16 values from seeded generators.

The shapes stand in for the multi-turn tool-use rollouts of the paper's
gpt-oss-20b policy (§4 and App. B, Tab. "hparams": GRPO with n = 8 trajectories
per task, 128k maximum sequence length; §3.2: each turn alternates generation
with a tool observation). The attention geometry (64 query heads, 8 KV heads,
head_dim 64, alternating full / 128-token sliding-window layers) is that of
gpt-oss-20b; the paper itself prints no attention shapes, no datasets are
read, and every number here is synthetic.

KV pool layout, shared by every consumer: ``[num_pages, H_kv, page_size, D]``
bf16, so one (page, kv head) block is ``page_size * D * 2`` contiguous bytes.
``seq_lens[r]`` is the KV length of row r *after* this step's append, and
``query_start_loc`` is the exclusive prefix sum of the per-row query counts.
A block-table entry of -1 marks a logical page that no query of the row can
see (sliding-window layers allocate only in-window pages).
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np
import torch

PAGE = 16
HEAD_DIM = 64


@dataclass
class Pool:
    """One paged KV pool and the block table that maps each row into it."""

    k_cache: torch.Tensor  # [num_pages, H_kv, page, D] bf16
    v_cache: torch.Tensor
    block_table: np.ndarray  # [B, max_pages_per_seq] int32, -1 = unallocated
    sliding_window: int  # window the pool was allocated for (0 = none)

    @property
    def num_pages(self) -> int:
        return int(self.k_cache.shape[0])


@dataclass
class Layer:
    """Per-layer inputs of one step: queries and the K/V rows to append."""

    q: torch.Tensor  # [T_q, H_q, D] bf16
    k_new: torch.Tensor  # [T_q, H_kv, D] bf16
    v_new: torch.Tensor
    pool: str  # key into Batch.pools
    sliding_window: int


@dataclass
class Batch:
    name: str
    seed: int
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    page_size: int
    softmax_scale: float
    seq_lens: np.ndarray  # [B] int32, KV length after the append
    query_start_loc: np.ndarray  # [B + 1] int32
    pools: dict
    layers: list
    group_of_row: np.ndarray | None = None  # GRPO group id per row, or None
    notes: dict = field(default_factory=dict)

    @property
    def num_seqs(self) -> int:
        return int(self.seq_lens.shape[0])

    @property
    def total_q(self) -> int:
        return int(self.query_start_loc[-1])

    @property
    def q_lens(self) -> np.ndarray:
        return np.diff(self.query_start_loc).astype(np.int32)


def _randn(shape, gen, device):
    return torch.randn(shape, generator=gen, device=device, dtype=torch.bfloat16)


def _log_uniform_int(rng, lo, hi, size):
    x = np.exp(rng.uniform(math.log(lo), math.log(hi), size=size))
    return np.clip(np.rint(x), lo, hi).astype(np.int64)


def build_batch(
    name: str,
    seed: int,
    seq_lens,
    q_lens,
    num_q_heads: int,
    num_kv_heads: int,
    *,
    head_dim: int = HEAD_DIM,
    page_size: int = PAGE,
    layer_windows=(0,),
    shared_prefix_pages=None,
    prompt_lens=None,
    group_of_row=None,
    device="cpu",
    peaked: bool = False,
    softmax_scale: float | None = None,
    pool_slack_pages: int = 0,
) -> Batch:
    """Allocate pools, block tables and values for explicit lengths.

    ``layer_windows[i]`` is the sliding window of layer i (0 = full context);
    layers with equal windows share one pool.  ``shared_prefix_pages[r]`` > 0
    makes row r reuse the physical pages of the first row of its group
    (``group_of_row``) for its first ``shared_prefix_pages[r]`` logical pages,
    as the G samples of a GRPO group share their prompt (full-context pools
    only).  ``prompt_lens`` lets the private page that follows the shared ones
    start with the same prompt-tail values in every member.
    """
    rng = np.random.Generator(np.random.PCG64(seed))
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    seq_lens = np.asarray(seq_lens, dtype=np.int64)
    q_lens = np.asarray(q_lens, dtype=np.int64)
    B = int(seq_lens.shape[0])
    assert q_lens.shape == (B,)
    assert np.all(q_lens >= 0) and np.all(q_lens <= seq_lens)
    qsl = np.zeros(B + 1, dtype=np.int64)
    qsl[1:] = np.cumsum(q_lens)
    max_pages = max(1, int(max((int(s) + page_size - 1) // page_size for s in seq_lens)))
    if shared_prefix_pages is None:
        shared_prefix_pages = np.zeros(B, dtype=np.int64)
    shared_prefix_pages = np.asarray(shared_prefix_pages, dtype=np.int64)

    pools = {}
    for w in sorted(set(int(w) for w in layer_windows)):
        bt = np.full((B, max_pages), -1, dtype=np.int64)
        # Logical pages each row needs: all of them for a full pool; for a
        # window pool only those covering keys [S - L - W + 1, S).
        owner = []  # (row, logical page) of every freshly allocated page
        shared_entries = []  # (row, logical page, row that owns the page)
        first_member = {}
        for r in range(B):
            S, L = int(seq_lens[r]), int(q_lens[r])
            hi = (S + page_size - 1) // page_size
            lo = 0 if w <= 0 else max(0, S - L - w + 1) // page_size
            nsh = int(shared_prefix_pages[r]) if w <= 0 else 0
            g = None if group_of_row is None else int(group_of_row[r])
            for lp in range(lo, hi):
                if nsh > 0 and lp < nsh and g in first_member:
                    shared_entries.append((r, lp, first_member[g]))
                else:
                    bt[r, lp] = len(owner)
                    owner.append((r, lp))
            if nsh > 0 and g not in first_member:
                first_member[g] = r
        num_pages = len(owner) + pool_slack_pages
        perm = rng.permutation(num_pages)
        phys = np.full((B, max_pages), -1, dtype=np.int64)
        alloc = bt >= 0
        phys[alloc] = perm[bt[alloc]]
        for r, lp, src in shared_entries:
            phys[r, lp] = phys[src, lp]
        shape = (num_pages, num_kv_heads, page_size, head_dim)
        k_cache = _randn(shape, gen, device)
        v_cache = _randn(shape, gen, device)
        if w <= 0 and prompt_lens is not None and group_of_row is not None:
            # The partial page after the shared ones holds the same prompt
            # tokens in every member (a private copy of the prompt tail).
            for r in range(B):
                g = int(group_of_row[r])
                src = first_member.get(g)
                nsh = int(shared_prefix_pages[r])
                tail = int(prompt_lens[r]) - nsh * page_size
                if src is None or src == r or tail <= 0 or nsh >= max_pages:
                    continue
                if phys[r, nsh] < 0 or phys[src, nsh] < 0:
                    continue
                dst_p, src_p = int(phys[r, nsh]), int(phys[src, nsh])
                k_cache[dst_p, :, :tail] = k_cache[src_p, :, :tail]
                v_cache[dst_p, :, :tail] = v_cache[src_p, :, :tail]
        pools[f"w{w}"] = Pool(k_cache, v_cache, phys.astype(np.int32), w)

    T = int(qsl[-1])
    layers = []
    for w in layer_windows:
        q = _randn((T, num_q_heads, head_dim), gen, device)
        k_new = _randn((T, num_kv_heads, head_dim), gen, device)
        v_new = _randn((T, num_kv_heads, head_dim), gen, device)
        layers.append(Layer(q, k_new, v_new, f"w{int(w)}", int(w)))

    if peaked:
        _make_peaked(layers, pools, seq_lens, q_lens, qsl, num_q_heads, num_kv_heads, page_size, rng)

    scale = 1.0 / math.sqrt(head_dim) if softmax_scale is None else float(softmax_scale)
    return Batch(
        name=name,
        seed=seed,
        num_q_heads=num_q_heads,
        num_kv_heads=num_kv_heads,
        head_dim=head_dim,
        page_size=page_size,
        softmax_scale=scale,
        seq_lens=seq_lens.astype(np.int32),
        query_start_loc=qsl.astype(np.int32),
        pools=pools,
        layers=layers,
        group_of_row=None if group_of_row is None else np.asarray(group_of_row, np.int32),
    )


def _make_peaked(layers, pools, seq_lens, q_lens, qsl, Hq, Hkv, page_size, rng):
    """Stress variant: scale Q by 4 (exact in bf16) and plant, for the first
    query of each row, a key equal to that query's (unscaled) vector, so the
    softmax is dominated by few keys and errors are not averaged away."""
    g = Hq // Hkv
    for layer in layers:
        pool = pools[layer.pool]
        bt = pool.block_table
        for r in range(len(seq_lens)):
            S, L = int(seq_lens[r]), int(q_lens[r])
            if L == 0:
                continue
            t0 = int(qsl[r])
            p = S - L  # position of the first query
            lo = 0 if layer.sliding_window <= 0 else max(0, p - layer.sliding_window + 1)
            j = int(rng.integers(lo, p + 1))
            if j >= S - L:
                continue  # would land on an appended slot (overwritten by the append)
            page = int(bt[r, j // page_size])
            for h in range(Hkv):
                pool.k_cache[page, h, j % page_size] = layer.q[t0, h * g]
        layer.q.mul_(4)


# ---------------------------------------------------------------------------
# The five workload configurations (shapes of gpt-oss-20b rollouts).
# ---------------------------------------------------------------------------


def config_tiny(seed=1001, device="cpu") -> Batch:
    """Tiny decode: 4 rows with KV lengths {17, 64, 129, 300}, 8 q / 2 kv
    heads, one query token each, block table a seeded page permutation."""
    return build_batch("tiny_decode", seed, [17, 64, 129, 300], [1, 1, 1, 1], 8, 2, device=device)


def config_decode(seed=1002, device="cpu") -> Batch:
    """Decode batch: 64 rows, KV lengths uniform in [2048, 16384], one query
    token each, 64 q / 8 kv heads."""
    rng = np.random.Generator(np.random.PCG64(seed + 7919))
    S = rng.integers(2048, 16384, size=64, endpoint=True)
    return build_batch("decode_b64", seed, S, np.ones(64, np.int64), 64, 8, device=device)


def config_mixed(seed=1003, device="cpu") -> Batch:
    """Mixed multi-turn batch: 256 rows with prior context uniform in
    [4096, 32768]; 224 rows decode one token, 32 rows (a seeded choice)
    append a tool-observation chunk of log-uniform length in [64, 2048]."""
    rng = np.random.Generator(np.random.PCG64(seed + 7919))
    B = 256
    prior = rng.integers(4096, 32768, size=B, endpoint=True)
    append_rows = rng.permutation(B)[:32]
    L = np.ones(B, np.int64)
    L[append_rows] = _log_uniform_int(rng, 64, 2048, 32)
    return build_batch("mixed_b256", seed, prior + L, L, 64, 8, device=device)


def config_long(seed=1004, device="cpu") -> Batch:
    """Long-horizon decode: 512 rows, KV lengths log-normal with median 12288
    (sigma 1, natural log), clipped to [512, 65536]; a seeded third of the
    rows (171) redrawn uniform in [49152, 65536]."""
    rng = np.random.Generator(np.random.PCG64(seed + 7919))
    B = 512
    S = np.clip(np.rint(np.exp(rng.normal(math.log(12288), 1.0, size=B))), 512, 65536).astype(np.int64)
    forced = rng.permutation(B)[:171]
    S[forced] = rng.integers(49152, 65536, size=171, endpoint=True)
    return build_batch("long_b512", seed, S, np.ones(B, np.int64), 64, 8, device=device)


def rollout_lengths(seed=1005, groups=48, group_size=8, append_frac=0.15):
    """Lengths of the GRPO rollout step: ``groups`` tasks x ``group_size``
    samples; prompt uniform in [1024, 8192] shared within a group, private
    continuation uniform in [0, 24576]; 15 % of rows (a seeded choice) append
    a chunk of log-uniform length in [64, 1024], the rest decode one token."""
    rng = np.random.Generator(np.random.PCG64(seed + 7919))
    B = groups * group_size
    group_of_row = np.repeat(np.arange(groups), group_size)
    prompt_g = rng.integers(1024, 8192, size=groups, endpoint=True)
    prompt = prompt_g[group_of_row]
    cont = rng.integers(0, 24576, size=B, endpoint=True)
    n_app = int(round(append_frac * B))
    app_rows = rng.permutation(B)[:n_app]
    L = np.ones(B, np.int64)
    L[app_rows] = _log_uniform_int(rng, 64, 1024, n_app)
    S = prompt + cont + L
    shared = prompt // PAGE
    return S, L, group_of_row, prompt, shared


def config_rollout(seed=1005, device="cpu", layers=24, window=128, groups=48, name=None) -> Batch:
    """Full rollout step: ``layers`` layers alternating sliding-window-128
    (even) and full-context (odd) attention over 48 GRPO groups x 8 rows.
    Full-context layers share one pool in which every group's full prompt
    pages are referenced by all 8 block tables; window layers share a second
    pool that holds only in-window pages."""
    S, L, grp, prompt, shared = rollout_lengths(seed, groups=groups)
    wins = [window if (i % 2 == 0) else 0 for i in range(layers)]
    b = build_batch(
        name or f"rollout_g{groups}x8",
        seed,
        S,
        L,
        64,
        8,
        layer_windows=wins,
        shared_prefix_pages=shared,
        prompt_lens=prompt,
        group_of_row=grp,
        device=device,
    )
    return b


def config_mixed_small(seed=1013, device="cpu") -> Batch:
    """The mixed batch's distributions at a quarter of its rows (64 rows, 8
    appending): a profiling case whose pool (~2 GB) is still far above L2."""
    rng = np.random.Generator(np.random.PCG64(seed + 7919))
    B = 64
    prior = rng.integers(4096, 32768, size=B, endpoint=True)
    append_rows = rng.permutation(B)[:8]
    L = np.ones(B, np.int64)
    L[append_rows] = _log_uniform_int(rng, 64, 2048, 8)
    return build_batch("mixed_b64", seed, prior + L, L, 64, 8, device=device)


def config_rollout_small(seed=1015, device="cpu") -> Batch:
    """The rollout step's distributions at 8 GRPO groups (64 rows, 10
    appending) and 4 layers (window, full, window, full): a profiling case
    for the window and full-context layers' kernels whose pools stay small."""
    return config_rollout(seed=seed, device=device, layers=4, groups=8, name="rollout_g8x8_l4")


CONFIGS = {
    "tiny": config_tiny,
    "decode": config_decode,
    "mixed": config_mixed,
    "mixed_small": config_mixed_small,
    "long": config_long,
    "rollout": config_rollout,
    "rollout_small": config_rollout_small,
}


def fuzz_batch(seed: int, device="cpu", max_len=300, max_chunk=80) -> Batch:
    """Small random batch: 1-9 rows, KV lengths in [1, max_len] with extra
    weight on page-boundary values, chunk lengths in [1, max_chunk], window in
    {0, 1, 16, 128, 1000}, GQA group in {1, 4, 8}."""
    rng = np.random.Generator(np.random.PCG64(seed))
    B = int(rng.integers(1, 10))
    special = [1, 15, 16, 17, 31, 32, 33, 48, 64, 127, 128, 129, max_len]
    S = np.array(
        [int(rng.choice(special)) if rng.random() < 0.4 else int(rng.integers(1, max_len + 1)) for _ in range(B)],
        np.int64,
    )
    L = np.array([1 if rng.random() < 0.5 else int(rng.integers(1, min(max_chunk, s) + 1)) for s in S], np.int64)
    Hkv = int(rng.choice([1, 2]))
    g = int(rng.choice([1, 4, 8]))
    W = int(rng.choice([0, 1, 16, 128, 1000]))
    return build_batch(f"fuzz{seed}", seed, S, L, Hkv * g, Hkv, layer_windows=(W,), device=device)


# ---------------------------------------------------------------------------
# Host copies for the oracle.
# ---------------------------------------------------------------------------


def to_host(t: torch.Tensor) -> np.ndarray:
    """bf16 tensor -> numpy uint16 array holding the same bits."""
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def host_inputs(batch: Batch, layer: int = 0) -> dict:
    """Every input of one layer as host numpy arrays (bf16 kept as uint16)."""
    lay = batch.layers[layer]
    pool = batch.pools[lay.pool]
    return dict(
        q=to_host(lay.q),
        k_new=to_host(lay.k_new),
        v_new=to_host(lay.v_new),
        k_cache=to_host(pool.k_cache),
        v_cache=to_host(pool.v_cache),
        block_table=pool.block_table.copy(),
        seq_lens=batch.seq_lens.copy(),
        query_start_loc=batch.query_start_loc.copy(),
        sliding_window=lay.sliding_window,
        softmax_scale=batch.softmax_scale,
        num_q_heads=batch.num_q_heads,
        num_kv_heads=batch.num_kv_heads,
        head_dim=batch.head_dim,
        page_size=batch.page_size,
    )


def host_rows(batch: Batch, rows, layer: int = 0) -> dict:
    """The inputs of a subset of rows as a self-contained host problem.

    Only the physical pages those rows reference are copied (device gather,
    then one device-to-host copy); the block table is renumbered into the
    compact pool.  Used to check sampled rows of workloads whose full pool is
    too large to copy.  Returns the host dict plus ``token_map``: for each
    query token of the compact problem, its index in the full batch.
    """
    lay = batch.layers[layer]
    pool = batch.pools[lay.pool]
    rows = np.asarray(sorted(set(int(r) for r in rows)), np.int64)
    bt = pool.block_table[rows]
    used = np.unique(bt[bt >= 0])
    remap = np.full(pool.num_pages, -1, np.int64)
    remap[used] = np.arange(used.shape[0])
    bt_c = np.where(bt >= 0, remap[np.maximum(bt, 0)], -1).astype(np.int32)
    idx = torch.as_tensor(used, device=pool.k_cache.device)
    qsl = batch.query_start_loc
    tok = np.concatenate([np.arange(qsl[r], qsl[r + 1]) for r in rows]).astype(np.int64)
    tok_t = torch.as_tensor(tok, device=lay.q.device)
    L = (qsl[rows + 1] - qsl[rows]).astype(np.int64)
    qsl_c = np.zeros(len(rows) + 1, np.int64)
    qsl_c[1:] = np.cumsum(L)
    return dict(
        q=to_host(lay.q.index_select(0, tok_t)),
        k_new=to_host(lay.k_new.index_select(0, tok_t)),
        v_new=to_host(lay.v_new.index_select(0, tok_t)),
        k_cache=to_host(pool.k_cache.index_select(0, idx)),
        v_cache=to_host(pool.v_cache.index_select(0, idx)),
        block_table=bt_c,
        seq_lens=batch.seq_lens[rows].copy(),
        query_start_loc=qsl_c.astype(np.int32),
        sliding_window=lay.sliding_window,
        softmax_scale=batch.softmax_scale,
        num_q_heads=batch.num_q_heads,
        num_kv_heads=batch.num_kv_heads,
        head_dim=batch.head_dim,
        page_size=batch.page_size,
        token_map=tok,
        rows=rows,
    )


def rope_table(max_position: int, head_dim: int = HEAD_DIM, base: float = 150000.0) -> np.ndarray:
    """A rotary-embedding table [max_position, head_dim] float32: for position
    p and i < head_dim / 2, cos(p * base^(-2i/D)) then sin(...). An input of
    the fused RoPE + KV append (engines precompute it per model); base 150000
    is gpt-oss's rotary base, without its long-context rescaling."""
    half = head_dim // 2
    inv = base ** (-np.arange(half, dtype=np.float64) * 2.0 / head_dim)
    ang = np.arange(max_position, dtype=np.float64)[:, None] * inv[None, :]
    return np.concatenate([np.cos(ang), np.sin(ang)], axis=1).astype(np.float32)
