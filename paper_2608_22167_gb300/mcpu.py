"""Thin ctypes binding of libmcpu.so (include/mcpu.h).

Argument marshalling only: every function forwards device pointers of torch
tensors, the sizes read from their shapes and the current CUDA stream to the
C entry point of the same name, and raises ``McpuError`` on a non-OK status.
No computation happens here and there is no fallback: if the library is
missing, importing this module fails.
"""
from __future__ import annotations

import ctypes
import os

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "_build", "libmcpu.so")

if not os.path.exists(LIB_PATH):
    raise ImportError(
        f"libmcpu.so not found at {LIB_PATH}; build it first with "
        "`python -c 'import __graft_entry__ as g; g.build()'` (needs nvcc)"
    )
_lib = ctypes.CDLL(LIB_PATH)

STATUS = {
    0: "MCPU_OK",
    1: "MCPU_ERR_INVALID_ARG",
    2: "MCPU_ERR_UNSUPPORTED",
    3: "MCPU_ERR_WORKSPACE_TOO_SMALL",
    4: "MCPU_ERR_CUDA",
    5: "MCPU_ERR_BAD_PAGE",
    6: "MCPU_ERR_BAD_LENGTHS",
    7: "MCPU_ERR_TIMEOUT",
    8: "MCPU_ERR_INTERNAL",
    9: "MCPU_ERR_POOL_EXHAUSTED",
    10: "MCPU_ERR_UNSUPPORTED_ROW",
}
FLAG_NO_CASCADE = 0x1
FLAG_MMA_SYNC_APPEND = 0x2
FLAG_SERIAL = 0x4
FLAG_HOST_OUT_DIRECT = 0x8

# Device status bits (first word of the workspace).
STATUS_BAD_PAGE = 1
STATUS_BAD_LENGTHS = 2
STATUS_TIMEOUT = 4
STATUS_PLAN_OVERFLOW = 8
STATUS_POOL_EXHAUSTED = 16
STATUS_UNSUPPORTED_ROW = 32


class McpuError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        name = STATUS.get(code, str(code))
        msg = _lib.mcpu_status_string(code).decode()
        if code == 4:
            msg += f", cudaError_t {int(_lib.mcpu_last_cuda_error())}"
        super().__init__(f"{where}: {name} ({msg})")


class Dims(ctypes.Structure):
    _fields_ = [
        ("num_seqs", ctypes.c_int32),
        ("total_q", ctypes.c_int32),
        ("max_pages_per_seq", ctypes.c_int32),
        ("num_pages", ctypes.c_int32),
        ("num_q_heads", ctypes.c_int32),
        ("num_kv_heads", ctypes.c_int32),
        ("head_dim", ctypes.c_int32),
        ("page_size", ctypes.c_int32),
    ]


class Options(ctypes.Structure):
    _fields_ = [("flags", ctypes.c_uint32), ("split_pages", ctypes.c_int32), ("phase_events", ctypes.c_void_p),
                ("sinks", ctypes.c_void_p)]


NUM_PHASE_EVENTS = 6


_P = ctypes.c_void_p
_lib.mcpu_workspace_size.argtypes = [ctypes.POINTER(Dims)]
_lib.mcpu_workspace_size.restype = ctypes.c_size_t
_lib.mcpu_kv_append.argtypes = [_P, _P, _P, _P, _P, _P, _P, ctypes.POINTER(Dims), _P, _P]
_lib.mcpu_kv_append.restype = ctypes.c_int
_lib.mcpu_paged_attention_forward.argtypes = [
    _P, _P, _P, _P, _P, _P, ctypes.c_int32, ctypes.c_float, ctypes.POINTER(Dims), _P, _P, _P, ctypes.c_size_t,
    ctypes.POINTER(Options), _P,
]
_lib.mcpu_paged_attention_forward.restype = ctypes.c_int
_lib.mcpu_paged_attention_forward_noalloc.argtypes = [
    _P, _P, _P, _P, _P, _P, ctypes.c_int32, ctypes.c_float, ctypes.POINTER(Dims), _P, _P, _P, _P,
]
_lib.mcpu_paged_attention_forward_noalloc.restype = ctypes.c_int
_lib.mcpu_rope_kv_append.argtypes = [_P, _P, _P, _P, _P, _P, _P, _P, _P, ctypes.c_int32, ctypes.POINTER(Dims), _P, _P]
_lib.mcpu_rope_kv_append.restype = ctypes.c_int
_lib.mcpu_grow_block_tables.argtypes = [_P, _P, ctypes.POINTER(Dims), _P, _P, _P, _P]
_lib.mcpu_grow_block_tables.restype = ctypes.c_int
_lib.mcpu_kv_append_fp8.argtypes = [_P, _P, _P, _P, _P, _P, ctypes.POINTER(Dims), _P, _P]
_lib.mcpu_kv_append_fp8.restype = ctypes.c_int
_lib.mcpu_paged_attention_forward_fp8.argtypes = [
    _P, _P, _P, _P, _P, ctypes.c_int32, ctypes.c_float, ctypes.POINTER(Dims), _P, _P, _P, ctypes.c_size_t,
    ctypes.POINTER(Options), _P,
]
_lib.mcpu_paged_attention_forward_fp8.restype = ctypes.c_int
_lib.mcpu_read_device_status.argtypes = [_P, _P, ctypes.POINTER(ctypes.c_int32)]
_lib.mcpu_read_device_status.restype = ctypes.c_int
_lib.mcpu_reset_device_status.argtypes = [_P, _P]
_lib.mcpu_reset_device_status.restype = ctypes.c_int
_lib.mcpu_selftest_wait_timeout.argtypes = [_P, _P, _P]
_lib.mcpu_selftest_wait_timeout.restype = ctypes.c_int
_lib.mcpu_selftest_append_abort.argtypes = [
    _P, _P, _P, _P, _P, _P, ctypes.c_float, ctypes.POINTER(Dims), _P, _P, _P, ctypes.c_size_t, ctypes.c_int32, _P, _P,
]
_lib.mcpu_selftest_append_abort.restype = ctypes.c_int
_lib.mcpu_status_string.argtypes = [ctypes.c_int]
_lib.mcpu_status_string.restype = ctypes.c_char_p
_lib.mcpu_abi_version.argtypes = []
_lib.mcpu_abi_version.restype = ctypes.c_int32
_lib.mcpu_last_cuda_error.argtypes = []
_lib.mcpu_last_cuda_error.restype = ctypes.c_int32
_lib.mcpu_host_stage_create.argtypes = [ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                                        ctypes.c_int32, ctypes.POINTER(ctypes.c_void_p)]
_lib.mcpu_host_stage_create.restype = ctypes.c_int
_lib.mcpu_host_stage_destroy.argtypes = [_P]
_lib.mcpu_host_stage_destroy.restype = ctypes.c_int
_lib.mcpu_host_stage_wait.argtypes = [_P, _P]
_lib.mcpu_host_stage_wait.restype = ctypes.c_int
_lib.mcpu_host_stage_sync.argtypes = [_P]
_lib.mcpu_host_stage_sync.restype = ctypes.c_int
_lib.mcpu_host_slice_rows.argtypes = [_P, ctypes.c_int32, ctypes.c_int32, _P]
_lib.mcpu_host_slice_rows.restype = ctypes.c_int32
_lib.mcpu_paged_attention_host.argtypes = [
    _P, _P, _P, _P, _P, _P, _P, _P, _P, ctypes.c_int32, ctypes.c_float, ctypes.POINTER(Dims), _P, _P, _P,
    ctypes.c_size_t, ctypes.POINTER(Options), ctypes.c_int32, _P,
]
_lib.mcpu_paged_attention_host.restype = ctypes.c_int
_lib.mcpu_paged_attention_host_fp8.argtypes = [
    _P, _P, _P, _P, _P, _P, _P, _P, ctypes.c_int32, ctypes.c_float, ctypes.POINTER(Dims), _P, _P, _P,
    ctypes.c_size_t, ctypes.POINTER(Options), ctypes.c_int32, _P,
]
_lib.mcpu_paged_attention_host_fp8.restype = ctypes.c_int

MAX_HOST_SLICES = 8
MAX_HOST_SLOTS = 4


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _check(code, where):
    if code != 0:
        raise McpuError(code, where)


def dims(q, k_cache, block_table, seq_lens) -> Dims:
    """mcpu_dims from tensor shapes: q [T, Hq, D], k_cache [P, Hkv, page, D],
    block_table [B, max_pages], seq_lens [B]."""
    return Dims(
        num_seqs=int(seq_lens.shape[0]),
        total_q=int(q.shape[0]),
        max_pages_per_seq=int(block_table.shape[1]),
        num_pages=int(k_cache.shape[0]),
        num_q_heads=int(q.shape[1]),
        num_kv_heads=int(k_cache.shape[1]),
        head_dim=int(q.shape[2]),
        page_size=int(k_cache.shape[2]),
    )


def mcpu_abi_version() -> int:
    return int(_lib.mcpu_abi_version())


def mcpu_last_cuda_error() -> int:
    return int(_lib.mcpu_last_cuda_error())


def mcpu_status_string(code: int) -> str:
    return _lib.mcpu_status_string(code).decode()


def mcpu_workspace_size(d: Dims) -> int:
    return int(_lib.mcpu_workspace_size(ctypes.byref(d)))


def mcpu_kv_append(k_new, v_new, k_cache, v_cache, block_table, seq_lens, query_start_loc, status_word,
                   stream=None):
    """status_word: a device int32 tensor (e.g. ``workspace[:4].view(torch.int32)``)."""
    d = Dims(
        num_seqs=int(seq_lens.shape[0]),
        total_q=int(k_new.shape[0]),
        max_pages_per_seq=int(block_table.shape[1]),
        num_pages=int(k_cache.shape[0]),
        num_q_heads=int(k_cache.shape[1]),
        num_kv_heads=int(k_cache.shape[1]),
        head_dim=int(k_cache.shape[3]),
        page_size=int(k_cache.shape[2]),
    )
    _check(
        _lib.mcpu_kv_append(_ptr(k_new), _ptr(v_new), _ptr(k_cache), _ptr(v_cache), _ptr(block_table),
                            _ptr(seq_lens), _ptr(query_start_loc), ctypes.byref(d), _ptr(status_word),
                            _stream(stream)),
        "mcpu_kv_append",
    )


def mcpu_rope_kv_append(q, k_new, v_new, k_cache, v_cache, block_table, seq_lens, query_start_loc, cos_sin,
                        status_word, stream=None):
    """Rotates q in place and writes rotated k_new / v_new into the pools;
    cos_sin: float32 device tensor [max_position, 64] (cos then sin)."""
    if cos_sin.dtype != torch.float32 or cos_sin.dim() != 2 or cos_sin.shape[1] != q.shape[2]:
        raise ValueError("cos_sin must be a float32 [max_position, head_dim] tensor")
    d = dims(q, k_cache, block_table, seq_lens)
    _check(
        _lib.mcpu_rope_kv_append(_ptr(q), _ptr(k_new), _ptr(v_new), _ptr(k_cache), _ptr(v_cache), _ptr(block_table),
                                 _ptr(seq_lens), _ptr(query_start_loc), _ptr(cos_sin), int(cos_sin.shape[0]),
                                 ctypes.byref(d), _ptr(status_word), _stream(stream)),
        "mcpu_rope_kv_append",
    )


def mcpu_grow_block_tables(block_table, seq_lens, free_pages, free_count, status_word, stream=None):
    """Fills every negative block-table entry a row needs for its seq_len with
    a page popped from the device stack free_pages[0:free_count] (int32
    tensors; free_count is a one-element device tensor, decremented)."""
    d = Dims(num_seqs=int(seq_lens.shape[0]), total_q=0, max_pages_per_seq=int(block_table.shape[1]), num_pages=0,
             num_q_heads=1, num_kv_heads=1, head_dim=64, page_size=16)
    _check(
        _lib.mcpu_grow_block_tables(_ptr(block_table), _ptr(seq_lens), ctypes.byref(d), _ptr(free_pages),
                                    _ptr(free_count), _ptr(status_word), _stream(stream)),
        "mcpu_grow_block_tables",
    )


def _options(num_q_heads, flags, split_pages, phase_events, sinks) -> Options:
    opts = Options(flags=int(flags), split_pages=int(split_pages), phase_events=None, sinks=None)
    if sinks is not None:
        if sinks.dtype != torch.float32 or sinks.numel() != num_q_heads or not sinks.is_cuda:
            raise ValueError("sinks must be a float32 CUDA tensor with one value per q head")
        opts.sinks = ctypes.c_void_p(sinks.data_ptr())
    if phase_events is not None:
        assert len(phase_events) == NUM_PHASE_EVENTS
        if any(e.cuda_event == 0 for e in phase_events):
            raise ValueError("torch creates a CUDA event at its first record(): record each phase event once "
                             "before passing it")
        arr = (ctypes.c_void_p * NUM_PHASE_EVENTS)(*[ctypes.c_void_p(e.cuda_event) for e in phase_events])
        opts.phase_events = ctypes.cast(arr, ctypes.c_void_p)
        opts._events = arr  # keep the array alive as long as the options
    return opts


def mcpu_paged_attention_forward(q, k_cache, v_cache, block_table, seq_lens, query_start_loc, sliding_window,
                                 softmax_scale, out, lse, workspace, flags=0, split_pages=0, stream=None,
                                 phase_events=None, sinks=None):
    """phase_events: optional list of NUM_PHASE_EVENTS torch.cuda.Event the
    call records around its kernels (see mcpu_options in include/mcpu.h);
    sinks: optional float32 device tensor [H_q] of attention-sink logits."""
    d = dims(q, k_cache, block_table, seq_lens)
    opts = _options(d.num_q_heads, flags, split_pages, phase_events, sinks)
    _check(
        _lib.mcpu_paged_attention_forward(
            _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(block_table), _ptr(seq_lens), _ptr(query_start_loc),
            int(sliding_window), float(softmax_scale), ctypes.byref(d), _ptr(out), _ptr(lse), _ptr(workspace),
            int(workspace.numel() * workspace.element_size()), ctypes.byref(opts), _stream(stream),
        ),
        "mcpu_paged_attention_forward",
    )


def mcpu_paged_attention_forward_noalloc(q, k_cache, v_cache, block_table, seq_lens, query_start_loc,
                                         sliding_window, softmax_scale, out, lse, status_word=None, stream=None):
    """The forward without a workspace (scratch in the library's own device
    memory); status_word: optional device int32 tensor for the status bits."""
    d = dims(q, k_cache, block_table, seq_lens)
    _check(
        _lib.mcpu_paged_attention_forward_noalloc(
            _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(block_table), _ptr(seq_lens), _ptr(query_start_loc),
            int(sliding_window), float(softmax_scale), ctypes.byref(d), _ptr(out), _ptr(lse), _ptr(status_word),
            _stream(stream),
        ),
        "mcpu_paged_attention_forward_noalloc",
    )


FP8_BLOCK_BYTES = 2176  # one (page, kv head) block: K codes, V codes (transposed), K and V scales


def new_fp8_pool(num_pages, num_kv_heads, device="cuda") -> torch.Tensor:
    """An (uninitialised) fp8 KV pool: uint8 [num_pages, H_kv, 2176]."""
    return torch.empty((num_pages, num_kv_heads, FP8_BLOCK_BYTES), dtype=torch.uint8, device=device)


def dims_fp8(q, kv8, block_table, seq_lens) -> Dims:
    """mcpu_dims for an fp8 pool kv8 [P, Hkv, 2176]."""
    if kv8.dim() != 3 or kv8.shape[2] != FP8_BLOCK_BYTES or kv8.dtype != torch.uint8:
        raise ValueError("kv8 must be a uint8 [num_pages, H_kv, 2176] tensor")
    return Dims(num_seqs=int(seq_lens.shape[0]), total_q=int(q.shape[0]), max_pages_per_seq=int(block_table.shape[1]),
                num_pages=int(kv8.shape[0]), num_q_heads=int(q.shape[1]), num_kv_heads=int(kv8.shape[1]),
                head_dim=int(q.shape[2]), page_size=16)


def mcpu_kv_append_fp8(k_new, v_new, kv8, block_table, seq_lens, query_start_loc, status_word, stream=None):
    """Quantizing KV append into an fp8 pool kv8 (uint8 [P, Hkv, 2176])."""
    d = dims_fp8(k_new, kv8, block_table, seq_lens)
    d.num_q_heads = d.num_kv_heads
    _check(
        _lib.mcpu_kv_append_fp8(_ptr(k_new), _ptr(v_new), _ptr(kv8), _ptr(block_table), _ptr(seq_lens),
                                _ptr(query_start_loc), ctypes.byref(d), _ptr(status_word), _stream(stream)),
        "mcpu_kv_append_fp8",
    )


def mcpu_paged_attention_forward_fp8(q, kv8, block_table, seq_lens, query_start_loc, sliding_window, softmax_scale,
                                     out, lse, workspace, flags=0, split_pages=0, stream=None, phase_events=None,
                                     sinks=None):
    """Decode-row attention over an fp8 pool (layout as mcpu_kv_append_fp8)."""
    d = dims_fp8(q, kv8, block_table, seq_lens)
    opts = _options(d.num_q_heads, flags, split_pages, phase_events, sinks)
    _check(
        _lib.mcpu_paged_attention_forward_fp8(
            _ptr(q), _ptr(kv8), _ptr(block_table), _ptr(seq_lens), _ptr(query_start_loc), int(sliding_window),
            float(softmax_scale), ctypes.byref(d), _ptr(out), _ptr(lse), _ptr(workspace),
            int(workspace.numel() * workspace.element_size()), ctypes.byref(opts), _stream(stream),
        ),
        "mcpu_paged_attention_forward_fp8",
    )


def mcpu_read_device_status(workspace, stream=None):
    """(mcpu status code, raw status bits) of the workspace's status word."""
    bits = ctypes.c_int32(0)
    code = _lib.mcpu_read_device_status(_ptr(workspace), _stream(stream), ctypes.byref(bits))
    return int(code), int(bits.value)


def mcpu_reset_device_status(workspace, stream=None):
    _check(_lib.mcpu_reset_device_status(_ptr(workspace), _stream(stream)), "mcpu_reset_device_status")


def mcpu_selftest_wait_timeout(workspace, report, stream=None):
    """Enqueues the timeout self-check: ``report`` is a device int64 tensor of
    4 entries (completing wait ok, never-completing wait ok, its duration in
    ns, the wait limit in ns); the status word of ``workspace`` gets the
    timeout bit when the wait gives up."""
    if report.dtype != torch.int64 or report.numel() < 4 or not report.is_contiguous():
        raise McpuError(1, "mcpu_selftest_wait_timeout")
    _check(_lib.mcpu_selftest_wait_timeout(_ptr(workspace), _ptr(report), _stream(stream)),
           "mcpu_selftest_wait_timeout")


def mcpu_selftest_append_abort(q, k_cache, v_cache, block_table, seq_lens, query_start_loc, softmax_scale, out, lse,
                               workspace, stall_role, report, stream=None):
    """Enqueues the append kernel's abort self-check as one CTA over this
    batch: role ``stall_role`` (0 softmax of tile A, 1 producer, 2 issuer of
    tile A) waits on a barrier nothing completes; ``report`` is a device int64
    tensor of 16 entries (final abort flag, each warp's exit time in ns, the
    stalled wait, the wait limit, TMEM freed)."""
    if report.dtype != torch.int64 or report.numel() < 16 or not report.is_cuda:
        raise McpuError(1, "mcpu_selftest_append_abort")
    d = dims(q, k_cache, block_table, seq_lens)
    _check(
        _lib.mcpu_selftest_append_abort(
            _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(block_table), _ptr(seq_lens), _ptr(query_start_loc),
            float(softmax_scale), ctypes.byref(d), _ptr(out), _ptr(lse), _ptr(workspace),
            workspace.numel() * workspace.element_size(), int(stall_role), _ptr(report), _stream(stream),
        ),
        "mcpu_selftest_append_abort",
    )


def new_workspace(d: Dims, device="cuda") -> torch.Tensor:
    """A zeroed workspace of the size mcpu_workspace_size(d) asks for."""
    n = mcpu_workspace_size(d)
    if n == 0:
        raise McpuError(1, "mcpu_workspace_size")
    return torch.zeros(n, dtype=torch.uint8, device=device)


def status_word(workspace) -> torch.Tensor:
    """The device int32 status word at the start of a workspace."""
    return workspace[:4].view(torch.int32)


# ---------------------------------------------------------------- host buffers
class HostStage:
    """Handle of an mcpu_host_stage: device staging for calls with host
    buffers (see mcpu_paged_attention_host). Keeps the host tensors of every
    call made since the last sync() alive."""

    def __init__(self, max_tokens, max_rows, num_q_heads, num_kv_heads, slots=2):
        h = ctypes.c_void_p()
        _check(_lib.mcpu_host_stage_create(int(max_tokens), int(max_rows), int(num_q_heads), int(num_kv_heads),
                                           int(slots), ctypes.byref(h)), "mcpu_host_stage_create")
        self.handle = h
        self._pending = []

    def close(self):
        if self.handle:
            _lib.mcpu_host_stage_destroy(self.handle)
            self.handle = None
            self._pending = []

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def mcpu_host_stage_create(max_tokens, max_rows, num_q_heads, num_kv_heads, slots=2) -> HostStage:
    return HostStage(max_tokens, max_rows, num_q_heads, num_kv_heads, slots)


def mcpu_host_stage_destroy(stage: HostStage):
    stage.close()


def mcpu_host_stage_wait(stage: HostStage, stream=None):
    _check(_lib.mcpu_host_stage_wait(stage.handle, _stream(stream)), "mcpu_host_stage_wait")


def mcpu_host_stage_sync(stage: HostStage):
    _check(_lib.mcpu_host_stage_sync(stage.handle), "mcpu_host_stage_sync")
    stage._pending = []


def _host_i32(t):
    if t.is_cuda or t.dtype != torch.int32 or not t.is_contiguous():
        raise ValueError("expected a contiguous int32 host tensor")
    return t


def mcpu_host_slice_rows(query_start_loc_host, slices):
    """Row boundaries [0, ..., B] of the slices mcpu_paged_attention_host uses."""
    qsl = _host_i32(query_start_loc_host)
    rb = (ctypes.c_int32 * (MAX_HOST_SLICES + 1))()
    n = int(_lib.mcpu_host_slice_rows(_ptr(qsl), int(qsl.numel()) - 1, int(slices), ctypes.cast(rb, _P)))
    return [int(rb[i]) for i in range(n + 1)] if n > 0 else []


def mcpu_paged_attention_host(stage, q_host, k_new_host, v_new_host, k_cache, v_cache, block_table, seq_lens_host,
                              query_start_loc_host, sliding_window, softmax_scale, out_host, lse_host, workspace,
                              flags=0, split_pages=0, slices=0, stream=None, sinks=None):
    """KV append and forward of one layer whose q / k_new / v_new and out /
    lse are host (CPU) tensors, page-locked for full copy speed; seq_lens
    and query_start_loc are int32 host tensors; pools, block table and
    workspace stay on the device. The outputs are complete after
    mcpu_host_stage_sync(stage) (or, on the device, after
    mcpu_host_stage_wait(stage, stream))."""
    for t in (q_host, k_new_host, v_new_host, out_host, lse_host):
        if t.is_cuda or not t.is_contiguous():
            raise ValueError("q / k_new / v_new / out / lse must be contiguous host tensors")
    sl, qsl = _host_i32(seq_lens_host), _host_i32(query_start_loc_host)
    d = dims(q_host, k_cache, block_table, sl)
    opts = _options(d.num_q_heads, flags, split_pages, None, sinks)
    _check(
        _lib.mcpu_paged_attention_host(
            stage.handle, _ptr(q_host), _ptr(k_new_host), _ptr(v_new_host), _ptr(k_cache), _ptr(v_cache),
            _ptr(block_table), _ptr(sl), _ptr(qsl), int(sliding_window), float(softmax_scale), ctypes.byref(d),
            _ptr(out_host), _ptr(lse_host), _ptr(workspace), int(workspace.numel() * workspace.element_size()),
            ctypes.byref(opts), int(slices), _stream(stream),
        ),
        "mcpu_paged_attention_host",
    )
    stage._pending.append((q_host, k_new_host, v_new_host, out_host, lse_host, sl, qsl, opts))


def mcpu_paged_attention_host_fp8(stage, q_host, k_new_host, v_new_host, kv8, block_table, seq_lens_host,
                                  query_start_loc_host, sliding_window, softmax_scale, out_host, lse_host, workspace,
                                  flags=0, split_pages=0, slices=0, stream=None, sinks=None):
    """mcpu_paged_attention_host over an fp8 pool kv8 [P, Hkv, 2176] (decode rows)."""
    for t in (q_host, k_new_host, v_new_host, out_host, lse_host):
        if t.is_cuda or not t.is_contiguous():
            raise ValueError("q / k_new / v_new / out / lse must be contiguous host tensors")
    sl, qsl = _host_i32(seq_lens_host), _host_i32(query_start_loc_host)
    d = dims_fp8(q_host, kv8, block_table, sl)
    opts = _options(d.num_q_heads, flags, split_pages, None, sinks)
    _check(
        _lib.mcpu_paged_attention_host_fp8(
            stage.handle, _ptr(q_host), _ptr(k_new_host), _ptr(v_new_host), _ptr(kv8), _ptr(block_table), _ptr(sl),
            _ptr(qsl), int(sliding_window), float(softmax_scale), ctypes.byref(d), _ptr(out_host), _ptr(lse_host),
            _ptr(workspace), int(workspace.numel() * workspace.element_size()), ctypes.byref(opts), int(slices),
            _stream(stream),
        ),
        "mcpu_paged_attention_host_fp8",
    )
    stage._pending.append((q_host, k_new_host, v_new_host, out_host, lse_host, sl, qsl, opts))
