"""Host-side model of a rollout stage that keeps the attention path fed.

The paper's rollout layer (§3.2; App. C) overlaps hundreds of multi-turn
trajectories: environments are acquired, trajectories generate tokens on the
GPU, stop to call a tool, wait for its observation, append it, and continue
until they finish; the G samples of a GRPO task share one prompt (§4). This
module is a seeded stand-in for that pipeline. It holds no model and no
arithmetic of the attention itself: it decides, step by step, which rows are
in the batch and with how many query tokens, and it owns the KV pages.

Per step every live trajectory is in one of four states:

* ``ACQUIRE``  waiting for its environment (not in the batch);
* ``PREFILL``  first step: the group leader appends the whole prompt, the
               other members append only their private tail page's tokens;
* ``DECODE``   one query token (the response grows by one);
* ``WAIT``     a tool call is running (not in the batch); when it returns,
               the next step appends the observation as one chunk (L > 1).

Pages come from a free list. A group's full prompt pages are written once
and referenced by all G block tables (reference-counted); the partial prompt
page and everything after it are private. Block tables grow in place as rows
grow; pages return to the free list when a trajectory finishes (shared pages
when the last member does). Rows of a group stay adjacent in the batch, so
the device planner can find their shared prefix.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

PAGE = 16
ACQUIRE, PREFILL, DECODE, WAIT, APPEND, DONE = range(6)


@dataclass
class SimConfig:
    num_pages: int = 1 << 16         # KV pool size in pages
    max_pages_per_seq: int = 2048    # block-table width (32768 tokens)
    max_live_groups: int = 6         # concurrency: groups of G trajectories alive at once
    group_size: int = 8              # G samples per task
    prompt_len: tuple = (256, 2048)  # uniform
    response_len: tuple = (8, 64)    # log-uniform tokens generated per turn
    observation_len: tuple = (32, 512)  # log-uniform tool-observation chunk
    tool_wait_steps: tuple = (1, 6)  # uniform steps a tool call takes
    acquire_steps: tuple = (0, 3)    # uniform steps to acquire an environment
    max_turns: tuple = (2, 5)        # uniform turns per trajectory
    max_len: int = 16384             # a trajectory stops at this length


@dataclass
class Trajectory:
    tid: int
    group: int
    member: int
    state: int
    length: int = 0                  # tokens in its KV cache (before this step's append)
    pages: list = field(default_factory=list)  # physical page of each logical page
    countdown: int = 0               # steps left in ACQUIRE / WAIT
    to_generate: int = 0             # tokens left in the current response
    pending: int = 0                 # tokens to append at the next step (prefill / observation)
    turns_left: int = 0


@dataclass
class StepBatch:
    """One step's batch: rows in batch order (groups adjacent)."""
    tids: np.ndarray          # [B] trajectory ids
    groups: np.ndarray        # [B] group ids
    seq_lens: np.ndarray      # [B] int32, KV length after this step's append
    q_lens: np.ndarray        # [B] int32, query tokens (1 = decode, > 1 = append chunk)
    block_table: np.ndarray   # [B, max_pages_per_seq] int32 (-1 past the row's pages)

    @property
    def query_start_loc(self) -> np.ndarray:
        return np.concatenate([[0], np.cumsum(self.q_lens)]).astype(np.int32)

    @property
    def num_seqs(self) -> int:
        return int(self.seq_lens.shape[0])

    @property
    def total_q(self) -> int:
        return int(self.q_lens.sum())


class PagePool:
    """Free list of physical pages with reference counts."""

    def __init__(self, num_pages: int, rng: np.random.Generator):
        self.free = list(rng.permutation(num_pages)[::-1])  # scattered, as a long-running pool is
        self.refs = np.zeros(num_pages, np.int32)

    def alloc(self) -> int:
        if not self.free:
            raise RuntimeError("KV pool exhausted")
        p = int(self.free.pop())
        self.refs[p] = 1
        return p

    def share(self, p: int):
        self.refs[p] += 1

    def release(self, p: int):
        self.refs[p] -= 1
        assert self.refs[p] >= 0
        if self.refs[p] == 0:
            self.free.append(p)

    @property
    def in_use(self) -> int:
        return int((self.refs > 0).sum())


class RolloutSim:
    def __init__(self, cfg: SimConfig, seed: int):
        self.cfg = cfg
        self.rng = np.random.Generator(np.random.PCG64(seed))
        self.pool = PagePool(cfg.num_pages, self.rng)
        self.trajs: dict[int, Trajectory] = {}
        self.next_tid = 0
        self.next_group = 0
        self.step_no = 0
        self.finished = 0
        self.generated = 0  # decode tokens produced so far

    # ------------------------------------------------------------ draws
    def _uniform(self, lohi) -> int:
        return int(self.rng.integers(lohi[0], lohi[1], endpoint=True))

    def _log_uniform(self, lohi) -> int:
        lo, hi = np.log(lohi[0]), np.log(lohi[1])
        return int(np.rint(np.exp(self.rng.uniform(lo, hi))))

    # ------------------------------------------------------------ groups
    def _admit_groups(self):
        live = {t.group for t in self.trajs.values()}
        while len(live) < self.cfg.max_live_groups:
            gid = self.next_group
            self.next_group += 1
            live.add(gid)
            prompt = self._uniform(self.cfg.prompt_len)
            wait = self._uniform(self.cfg.acquire_steps)
            for m in range(self.cfg.group_size):
                t = Trajectory(self.next_tid, gid, m, ACQUIRE, countdown=wait, pending=prompt,
                               turns_left=self._uniform(self.cfg.max_turns))
                self.trajs[t.tid] = t
                self.next_tid += 1

    def _leader(self, gid) -> Trajectory | None:
        for t in self.trajs.values():
            if t.group == gid and t.member == 0:
                return t
        return None

    # ------------------------------------------------------------ pages
    def _grow(self, t: Trajectory, new_len: int):
        need = (new_len + PAGE - 1) // PAGE
        if need > self.cfg.max_pages_per_seq:
            raise RuntimeError("trajectory longer than the block table")
        while len(t.pages) < need:
            t.pages.append(self.pool.alloc())

    def _finish(self, t: Trajectory):
        for p in t.pages:
            self.pool.release(p)
        t.pages = []
        t.state = DONE
        self.finished += 1

    # ------------------------------------------------------------ step
    def step(self) -> StepBatch:
        """Advance every trajectory by one step and return the batch of the
        rows that run on the GPU in this step."""
        cfg = self.cfg
        self._admit_groups()
        rows = []  # (group, member, traj, q_len)
        # prompt sharing must be set up before members build their tables
        for t in sorted(self.trajs.values(), key=lambda x: (x.group, x.member)):
            if t.state == ACQUIRE:
                if t.countdown > 0:
                    t.countdown -= 1
                    continue
                t.state = PREFILL
            if t.state == PREFILL:
                prompt = t.pending
                full = prompt // PAGE
                if t.member == 0:
                    self._grow(t, prompt)
                    q_len = prompt
                else:
                    lead = self._leader(t.group)
                    assert lead is not None and len(lead.pages) >= full
                    for p in lead.pages[:full]:
                        self.pool.share(p)
                    t.pages = list(lead.pages[:full])
                    self._grow(t, prompt)
                    q_len = prompt - full * PAGE  # the private tail page only
                t.length = prompt
                t.pending = 0
                t.to_generate = self._log_uniform(cfg.response_len)
                t.state = DECODE
                if q_len > 0:
                    rows.append((t.group, t.member, t, q_len, prompt))
                continue
            if t.state == WAIT:
                if t.countdown > 0:
                    t.countdown -= 1
                    continue
                t.state = APPEND
            if t.state == APPEND:
                L = min(t.pending, cfg.max_len - t.length)
                t.pending = 0
                if L > 0:
                    self._grow(t, t.length + L)
                    t.length += L
                    rows.append((t.group, t.member, t, L, t.length))
                t.to_generate = self._log_uniform(cfg.response_len)
                t.state = DECODE
                continue
            if t.state == DECODE:
                if t.length >= cfg.max_len:
                    self._finish(t)
                    continue
                self._grow(t, t.length + 1)
                t.length += 1
                self.generated += 1
                rows.append((t.group, t.member, t, 1, t.length))
                t.to_generate -= 1
                if t.to_generate <= 0:
                    t.turns_left -= 1
                    if t.turns_left <= 0:
                        t.state = DONE  # finishes after this step's token
                    else:
                        t.state = WAIT
                        t.countdown = self._uniform(cfg.tool_wait_steps)
                        t.pending = self._log_uniform(cfg.observation_len)
        # the batch (groups adjacent, members in order)
        rows.sort(key=lambda r: (r[0], r[1]))
        B = len(rows)
        bt = np.full((B, cfg.max_pages_per_seq), -1, np.int32)
        for i, (_, _, t, _, S) in enumerate(rows):
            bt[i, :len(t.pages)] = t.pages
        batch = StepBatch(
            tids=np.array([r[2].tid for r in rows], np.int64),
            groups=np.array([r[0] for r in rows], np.int64),
            seq_lens=np.array([r[4] for r in rows], np.int32),
            q_lens=np.array([r[3] for r in rows], np.int32),
            block_table=bt,
        )
        # trajectories that finished with this step's token leave now
        for t in list(self.trajs.values()):
            if t.state == DONE:
                if t.pages:
                    self._finish(t)
                del self.trajs[t.tid]
        self.step_no += 1
        return batch
