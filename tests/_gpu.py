"""Helpers shared by the GPU tests: run a batch through the C ABI and
compare with the oracle at the stated tolerances.

Tolerances (floating point): out max |gpu - oracle| <= 2e-2 and
max |gpu - oracle| / max |oracle| <= 1e-2 per checked set (elementwise
relative error is meaningless for outputs near zero: long-context outputs are
averages of many N(0,1) rows), lse max abs <= 1e-3. KV append: bit-exact.
"""
from __future__ import annotations

import numpy as np
import torch

import oracle
import workloads as W
from paper_2608_22167_gb300 import mcpu

OUT_ABS = 2e-2
OUT_REL = 1e-2
LSE_ABS = 1e-3


class Run:
    """Device copies of one layer of a batch plus the outputs of one call."""

    def __init__(self, batch: W.Batch, layer: int = 0, device="cuda"):
        self.batch = batch
        self.layer = layer
        lay = batch.layers[layer]
        pool = batch.pools[lay.pool]
        dev = torch.device(device)
        self.q = lay.q.to(dev)
        self.k_new = lay.k_new.to(dev)
        self.v_new = lay.v_new.to(dev)
        self.kc = pool.k_cache.to(dev)
        self.vc = pool.v_cache.to(dev)
        if self.kc.data_ptr() == pool.k_cache.data_ptr():  # already on the device: keep the input intact
            self.kc = self.kc.clone()
            self.vc = self.vc.clone()
        self.bt = torch.from_numpy(pool.block_table).to(dev)
        self.sl = torch.from_numpy(batch.seq_lens).to(dev)
        self.qsl = torch.from_numpy(batch.query_start_loc).to(dev)
        self.window = lay.sliding_window
        self.dims = mcpu.dims(self.q, self.kc, self.bt, self.sl)
        self.ws = mcpu.new_workspace(self.dims, dev)
        self.out = torch.full_like(self.q, float("nan"))
        self.lse = torch.full(self.q.shape[:2], float("nan"), dtype=torch.float32, device=dev)

    def append(self):
        mcpu.mcpu_kv_append(self.k_new, self.v_new, self.kc, self.vc, self.bt, self.sl, self.qsl,
                            mcpu.status_word(self.ws))

    def forward(self, flags=0, split_pages=0, sinks=None):
        """sinks: optional numpy float32 [H_q] attention-sink logits."""
        sk = None if sinks is None else torch.from_numpy(np.asarray(sinks, np.float32)).to(self.q.device)
        mcpu.mcpu_paged_attention_forward(self.q, self.kc, self.vc, self.bt, self.sl, self.qsl, self.window,
                                          self.batch.softmax_scale, self.out, self.lse, self.ws, flags=flags,
                                          split_pages=split_pages, sinks=sk)

    def status(self):
        return mcpu.mcpu_read_device_status(self.ws)

    def header(self):
        h = self.ws[:32].view(torch.int32).cpu().numpy()
        return dict(status=int(h[0]), n_decode=int(h[1]), n_cascade=int(h[2]), n_append=int(h[3]),
                    n_merge=int(h[4]), split_pages=int(h[5]), n_parts=int(h[6]))

    def out_host(self):
        return self.out.float().cpu().numpy(), self.lse.cpu().numpy()


def oracle_full(batch: W.Batch, layer: int = 0, sinks=None):
    """Oracle outputs of a whole (small) layer, append applied first."""
    h = W.host_inputs(batch, layer)
    kc, vc = oracle.kv_append(h["k_new"], h["v_new"], h["k_cache"], h["v_cache"], h["block_table"],
                              h["seq_lens"], h["query_start_loc"])
    out, lse = oracle.paged_attention(h["q"], kc, vc, h["block_table"], h["seq_lens"], h["query_start_loc"],
                                      h["sliding_window"], h["softmax_scale"], sinks=sinks)
    return oracle.bf16_bits_to_float(out), lse, (kc, vc)


def oracle_sampled(batch: W.Batch, rows, n_per_row: int, rng, layer: int = 0, sinks=None):
    """Oracle at sampled (token, head) pairs of the given rows: returns
    (token indices in the batch, heads, out [n, D], lse [n])."""
    h = W.host_rows(batch, rows, layer)
    kc, vc = oracle.kv_append(h["k_new"], h["v_new"], h["k_cache"], h["v_cache"], h["block_table"],
                              h["seq_lens"], h["query_start_loc"])
    qsl = h["query_start_loc"]
    toks, heads = [], []
    for i in range(len(h["rows"])):
        t0, t1 = int(qsl[i]), int(qsl[i + 1])
        if t1 == t0:
            continue
        # always the first and last token of the row, then random ones
        cand = [t0, t1 - 1] + list(rng.integers(t0, t1, size=max(0, n_per_row - 2)))
        for t in cand[:n_per_row]:
            toks.append(int(t))
            heads.append(int(rng.integers(0, batch.num_q_heads)))
    toks = np.asarray(toks, np.int64)
    heads = np.asarray(heads, np.int32)
    out, lse = oracle.paged_attention_sampled(h["q"], kc, vc, h["block_table"], h["seq_lens"], qsl,
                                              h["sliding_window"], h["softmax_scale"], toks, heads, sinks=sinks)
    return h["token_map"][toks], heads, oracle.bf16_bits_to_float(out), lse


def assert_parity(got_out, got_lse, ref_out, ref_lse, what=""):
    got_out = np.asarray(got_out, np.float64)
    ref_out = np.asarray(ref_out, np.float64)
    assert np.all(np.isfinite(got_out)), f"{what}: non-finite outputs"
    err = np.abs(got_out - ref_out)
    max_abs = float(err.max()) if err.size else 0.0
    scale = float(np.abs(ref_out).max()) if err.size else 1.0
    rel = max_abs / max(scale, 1e-30)
    fin = np.isfinite(ref_lse)
    assert np.array_equal(fin, np.isfinite(got_lse)), f"{what}: lse finiteness differs"
    lse_err = float(np.abs(np.asarray(got_lse)[fin] - ref_lse[fin]).max()) if fin.any() else 0.0
    assert max_abs <= OUT_ABS, f"{what}: max abs err {max_abs:.3e}"
    assert rel <= OUT_REL, f"{what}: norm-relative err {rel:.3e}"
    assert lse_err <= LSE_ABS, f"{what}: lse abs err {lse_err:.3e}"
    return max_abs, rel, lse_err


# ------------------------------------------------------------ fp8 pools


def oracle_quantize_pool(k_bits, v_bits):
    """fp8 pools (codes [P, Hkv, 16, D] uint8 both, scales [P, Hkv, 16]) of
    whole bf16 pools, quantized by the oracle: every page is appended as one
    16-token row."""
    P, H, page, D = k_bits.shape
    tok = lambda x: np.ascontiguousarray(np.asarray(x).transpose(0, 2, 1, 3).reshape(P * page, H, D))  # noqa: E731
    z8 = np.zeros((P, H, page, D), np.uint8)
    zs = np.zeros((P, H, page), np.float32)
    bt = np.arange(P, dtype=np.int32)[:, None]
    sl = np.full(P, page, np.int32)
    qsl = (np.arange(P + 1, dtype=np.int32) * page)
    return oracle.kv_append_fp8(tok(k_bits), tok(v_bits), z8, z8, zs, zs, bt, sl, qsl)


def _fp8_v_order():
    """Byte position, inside the V area of a block, of (dim d, key j): the
    MMA-fragment order of the ABI (half h, lane 4r + c, word j', byte i)."""
    pos = np.empty((64, 16), np.int64)
    for d in range(64):
        mt, hf, r = d >> 4, (d >> 3) & 1, d & 7
        for key in range(16):
            c, i = key >> 2, key & 3
            pos[d, key] = (mt >> 1) * 512 + (4 * r + c) * 16 + 4 * ((mt & 1) * 2 + hf) + i
    return pos


def _fp8_scale_order():
    """Float index, inside the scale area, of the K scale of key j (the V
    scale sits two floats later): 16 bytes per r = 2 (j / 4) + j % 2."""
    j = np.arange(16)
    return 4 * (2 * (j >> 2) + (j & 1)) + ((j >> 1) & 1)


def to_fp8_blocks(k8, v8, ks, vs):
    """Oracle arrays (codes [P, Hkv, 16, D], scales [P, Hkv, 16]) -> the
    ABI's pool of 2176-byte blocks [P, Hkv, 2176]."""
    P, H, page, D = k8.shape
    blk = np.zeros((P, H, 2176), np.uint8)
    blk[..., :1024] = np.asarray(k8).reshape(P, H, page * D)
    vpos = _fp8_v_order()  # [D, 16]
    vt = np.asarray(v8).transpose(0, 1, 3, 2)  # [P, H, D, 16]
    varea = np.zeros((P, H, 1024), np.uint8)
    varea[..., vpos.reshape(-1)] = vt.reshape(P, H, -1)
    blk[..., 1024:2048] = varea
    sidx = _fp8_scale_order()
    sc = np.zeros((P, H, 32), np.float32)
    sc[..., sidx] = ks
    sc[..., sidx + 2] = vs
    blk[..., 2048:2176] = sc.view(np.uint8).reshape(P, H, 128)
    return blk


def from_fp8_blocks(blk):
    """Inverse of to_fp8_blocks."""
    blk = np.asarray(blk)
    P, H, _ = blk.shape
    k8 = blk[..., :1024].reshape(P, H, 16, 64)
    vpos = _fp8_v_order()
    v8 = blk[..., 1024:2048][..., vpos.reshape(-1)].reshape(P, H, 64, 16).transpose(0, 1, 3, 2)
    sc = np.ascontiguousarray(blk[..., 2048:2176]).view(np.float32).reshape(P, H, 32)
    sidx = _fp8_scale_order()
    return np.ascontiguousarray(k8), np.ascontiguousarray(v8), sc[..., sidx].copy(), sc[..., sidx + 2].copy()


class Fp8Run:
    """A decode batch on fp8 pools: the prior context quantized by the oracle
    and uploaded, then this step's rows appended on the device by
    mcpu_kv_append_fp8 (checked bit for bit against the oracle's append)."""

    def __init__(self, batch: W.Batch, layer: int = 0, device="cuda", garbage_slots=False):
        self.batch = batch
        self.layer = layer
        h = W.host_inputs(batch, layer)
        self.h = h
        k8, v8, ks, vs = oracle_quantize_pool(h["k_cache"], h["v_cache"])
        if garbage_slots:
            # slots no row can see hold NaN codes and NaN scales
            vis = np.zeros(ks.shape[0:1] + ks.shape[2:], bool)  # [P, 16]
            bt, sl = h["block_table"], h["seq_lens"]
            for r in range(len(sl)):
                for j in range(int(sl[r])):
                    vis[bt[r, j // 16], j % 16] = True
            hide = ~vis
            k8 = k8.copy(); v8 = v8.copy(); ks = ks.copy(); vs = vs.copy()
            k8.transpose(0, 2, 1, 3)[hide] = 0x7F
            v8.transpose(0, 2, 1, 3)[hide] = 0xFF
            ks.transpose(0, 2, 1)[hide] = np.nan
            vs.transpose(0, 2, 1)[hide] = np.nan
        self.before = (k8, v8, ks, vs)
        dev = torch.device(device)
        lay = batch.layers[layer]
        self.q = lay.q.to(dev)
        self.k_new = lay.k_new.to(dev)
        self.v_new = lay.v_new.to(dev)
        self.kv8 = torch.from_numpy(to_fp8_blocks(k8, v8, ks, vs)).to(dev)
        pool = batch.pools[lay.pool]
        self.bt = torch.from_numpy(pool.block_table).to(dev)
        self.sl = torch.from_numpy(batch.seq_lens).to(dev)
        self.qsl = torch.from_numpy(batch.query_start_loc).to(dev)
        self.window = lay.sliding_window
        self.dims = mcpu.dims_fp8(self.q, self.kv8, self.bt, self.sl)
        self.ws = mcpu.new_workspace(self.dims, dev)
        self.out = torch.full_like(self.q, float("nan"))
        self.lse = torch.full(self.q.shape[:2], float("nan"), dtype=torch.float32, device=dev)

    def append(self):
        mcpu.mcpu_kv_append_fp8(self.k_new, self.v_new, self.kv8, self.bt, self.sl, self.qsl,
                                mcpu.status_word(self.ws))

    def oracle_append(self):
        h = self.h
        return oracle.kv_append_fp8(h["k_new"], h["v_new"], *self.before, h["block_table"], h["seq_lens"],
                                    h["query_start_loc"])

    def forward(self, flags=0, split_pages=0, sinks=None):
        sk = None if sinks is None else torch.from_numpy(np.asarray(sinks, np.float32)).to(self.q.device)
        mcpu.mcpu_paged_attention_forward_fp8(self.q, self.kv8, self.bt, self.sl, self.qsl, self.window,
                                              self.batch.softmax_scale, self.out, self.lse, self.ws, flags=flags,
                                              split_pages=split_pages, sinks=sk)

    def status(self):
        return mcpu.mcpu_read_device_status(self.ws)

    def header(self):
        hd = self.ws[:32].view(torch.int32).cpu().numpy()
        return dict(status=int(hd[0]), n_decode=int(hd[1]), n_cascade=int(hd[2]), n_append=int(hd[3]),
                    n_merge=int(hd[4]), split_pages=int(hd[5]), n_parts=int(hd[6]))

    def pools_host(self):
        """The device pool as oracle arrays (k8, v8, k_scale, v_scale)."""
        return from_fp8_blocks(self.kv8.cpu().numpy())

    def out_host(self):
        return self.out.float().cpu().numpy(), self.lse.cpu().numpy()
