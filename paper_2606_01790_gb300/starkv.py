"""Thin Python binding of the C ABI in ``include/starkv.h`` (ctypes).

Argument marshalling only: every step of the compression stage runs in the
CUDA kernels of ``libstarkv.so``.  Tensors are torch tensors (device memory for
the device calls, host memory for ``step_host``); their data pointers are
handed to the library unchanged.  There is no fallback: if the library is not
built, importing the first call raises.
"""
from __future__ import annotations

import ctypes as C
from dataclasses import dataclass, fields
from pathlib import Path
from typing import List, Optional, Sequence

import numpy as np
import torch

LIB_PATH = Path(__file__).resolve().parent / "libstarkv.so"

OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_CUDA, ERR_TIMEOUT, ERR_NOMEM, ERR_DEVICE = range(7)

ABI_FUNCTIONS = [
    "starkv_default_config", "starkv_init_state", "starkv_reset_seq", "starkv_destroy_state",
    "starkv_get_config", "starkv_workspace_bytes", "starkv_score_layer", "starkv_select",
    "starkv_compact", "starkv_step", "starkv_step_host", "starkv_check_device_error",
    "starkv_set_wait_limit", "starkv_set_timing", "starkv_kernel_times", "starkv_last_error",
    "starkv_score_layer_noalloc", "starkv_selftest_wait", "starkv_slot_state_bytes", "starkv_export_slot",
    "starkv_import_slot", "starkv_window_attention",
]

KERNELS = ["score_lse", "score_accum", "pool", "calibrate", "compact", "attention", "attn_combine"]


SELECT_GLOBAL, SELECT_PER_HEAD = 0, 1   # starkv_config.select_mode


class StarkvError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"starkv status {status}: {msg}")
        self.status = status


class CConfig(C.Structure):
    _fields_ = [(n, C.c_int32) for n in (
        "n_layers", "n_heads", "n_kv_heads", "head_dim", "window", "grid_rows", "grid_cols",
        "pool_kernel", "mi_bins", "mi_grid", "n_warmup", "n_ramp", "max_seqs")] + \
        [(n, C.c_float) for n in (
            "lambda_", "tau", "rho_mi", "rho_t", "delta", "d_min", "t_min", "t_max", "eps", "eps_h")] + \
        [(n, C.c_int32) for n in ("select_mode", "decay_mode", "aeb_mode", "mi_span")]


class CSeq(C.Structure):
    _fields_ = [("k", C.c_void_p), ("v", C.c_void_p), ("q", C.c_void_p), ("meta", C.c_void_p),
                ("meta_layer_stride", C.c_int64), ("L", C.c_int32), ("cur_frame", C.c_int32),
                ("budget", C.c_int32), ("slot", C.c_int32), ("k_out", C.c_void_p),
                ("v_out", C.c_void_p), ("meta_out", C.c_void_p), ("idx", C.c_void_p),
                ("S", C.c_void_p), ("score", C.c_void_p), ("stats", C.c_void_p),
                ("meta_group_stride", C.c_int64), ("lse", C.c_void_p), ("attn_o", C.c_void_p),
                ("attn_lse", C.c_void_p)]


_lib: Optional[C.CDLL] = None


class CSlotHeader(C.Structure):
    """``starkv_slot_header``: the first 32 bytes of an exported slot state."""
    _fields_ = [("magic", C.c_uint32), ("version", C.c_uint32), ("n_layers", C.c_int32),
                ("n_kv_heads", C.c_int32), ("grid_rows", C.c_int32), ("grid_cols", C.c_int32),
                ("reserved", C.c_uint32 * 2)]


SLOT_MAGIC = 0x31564B53


def slot_state_bytes_for(n_layers: int, G: int, RC: int) -> int:
    """STARKV_SLOT_STATE_BYTES of the header."""
    return C.sizeof(CSlotHeader) + ((n_layers * 4 + 7) & ~7) + n_layers * G * 8 + n_layers * G * RC * 4


def lib() -> C.CDLL:
    """The loaded library (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not LIB_PATH.exists():
            raise RuntimeError(f"{LIB_PATH} is missing: build it with __graft_entry__.build()")
        L = C.CDLL(str(LIB_PATH))
        st = C.c_void_p
        for name in ("starkv_score_layer", "starkv_select", "starkv_compact"):
            getattr(L, name).argtypes = [st, C.c_int32, C.POINTER(CSeq), C.c_int32, C.c_void_p,
                                         C.c_size_t, C.c_void_p]
        for name in ("starkv_step", "starkv_step_host", "starkv_window_attention"):
            getattr(L, name).argtypes = [st, C.POINTER(CSeq), C.c_int32, C.c_void_p, C.c_size_t,
                                         C.c_void_p]
        L.starkv_score_layer_noalloc.argtypes = [st, C.c_int32, C.POINTER(CSeq), C.c_int32, C.c_void_p]
        L.starkv_default_config.argtypes = [C.POINTER(CConfig)]
        L.starkv_default_config.restype = None
        L.starkv_init_state.argtypes = [C.POINTER(CConfig), C.POINTER(C.c_void_p), C.c_void_p]
        L.starkv_reset_seq.argtypes = [st, C.c_int32, C.c_void_p]
        L.starkv_destroy_state.argtypes = [st]
        L.starkv_get_config.argtypes = [st, C.POINTER(CConfig)]
        L.starkv_workspace_bytes.argtypes = [st, C.POINTER(CSeq), C.c_int32, C.c_int32,
                                             C.POINTER(C.c_size_t)]
        L.starkv_check_device_error.argtypes = [st, C.c_void_p]
        L.starkv_set_wait_limit.argtypes = [st, C.c_uint64]
        L.starkv_selftest_wait.argtypes = [st, C.c_uint64, C.c_void_p]
        L.starkv_slot_state_bytes.argtypes = [st, C.POINTER(C.c_size_t)]
        L.starkv_export_slot.argtypes = [st, C.c_int32, C.c_void_p, C.c_size_t, C.c_void_p]
        L.starkv_import_slot.argtypes = [st, C.c_int32, C.c_void_p, C.c_size_t, C.c_void_p]
        L.starkv_set_timing.argtypes = [st, C.c_int32]
        L.starkv_kernel_times.argtypes = [st, C.POINTER(C.c_int64), C.POINTER(C.c_float)]
        L.starkv_last_error.argtypes = []
        L.starkv_last_error.restype = C.c_char_p
        for name in ABI_FUNCTIONS:
            if name not in ("starkv_default_config", "starkv_last_error"):
                getattr(L, name).restype = C.c_int
        _lib = L
    return _lib


def _check(status: int) -> None:
    if status != OK:
        raise StarkvError(status, lib().starkv_last_error().decode())


@dataclass
class Config:
    """Mirror of ``starkv_config`` (defaults: ``starkv_default_config``)."""

    n_layers: int = 28
    n_heads: int = 28
    n_kv_heads: int = 4
    head_dim: int = 128
    window: int = 32
    grid_rows: int = 52
    grid_cols: int = 52
    pool_kernel: int = 5
    mi_bins: int = 8
    mi_grid: int = 8
    n_warmup: int = 5
    n_ramp: int = 10
    max_seqs: int = 1
    lambda_: float = 0.5
    tau: float = 1.0
    rho_mi: float = 0.9
    rho_t: float = 0.9
    delta: float = 0.2
    d_min: float = 0.1
    t_min: float = 0.95
    t_max: float = 1.05
    eps: float = 1e-6
    eps_h: float = 1e-12
    select_mode: int = 0    # SELECT_GLOBAL (the paper's) or SELECT_PER_HEAD
    decay_mode: int = 0     # 0 exponential (Eq. 9), 1 linear, 2 power law (readings)
    aeb_mode: int = 0       # 0 entropy, 1 peak confidence (reading)
    mi_span: int = 0        # 0 every historical visual token, 1 the newest frame's

    def to_c(self) -> CConfig:
        c = CConfig()
        for f in fields(self):
            setattr(c, f.name, getattr(self, f.name))
        return c

    @staticmethod
    def default() -> "Config":
        c = CConfig()
        lib().starkv_default_config(C.byref(c))
        return Config(**{f.name: getattr(c, f.name) for f in fields(Config)})


def stats_stride(n_kv_heads: int) -> int:
    """Floats per layer in a stats buffer (``STARKV_STATS_STRIDE``)."""
    return 8 + 6 * n_kv_heads


def sel_rows(cfg: "Config") -> int:
    """Rows of idx / score / meta_out per layer: 1 (global selection) or G (per KV head)."""
    return cfg.n_kv_heads if cfg.select_mode == SELECT_PER_HEAD else 1


def pack_meta(is_visual, frame, row, col) -> np.ndarray:
    """Token metadata words of the ABI: bit 31 visual, 20..30 frame, 10..19 row, 0..9 col."""
    v = np.asarray(is_visual).astype(np.uint32) != 0
    f = np.asarray(frame).astype(np.uint32)
    r = np.asarray(row).astype(np.uint32)
    c = np.asarray(col).astype(np.uint32)
    if (f > 2047).any() or (r > 1023).any() or (c > 1023).any():
        raise ValueError("frame / row / col out of the metadata word's range")
    out = (v.astype(np.uint32) << np.uint32(31)) | (f << np.uint32(20)) | (r << np.uint32(10)) | c
    return np.where(v, out, np.uint32(0)).astype(np.uint32)


def unpack_meta(words: np.ndarray):
    w = np.asarray(words).astype(np.uint32)
    return ((w >> 31) & 1).astype(np.int32), ((w >> 20) & 0x7FF).astype(np.int32), \
        ((w >> 10) & 0x3FF).astype(np.int32), (w & 0x3FF).astype(np.int32)


def meta_tensor(words: np.ndarray) -> torch.Tensor:
    """uint32 metadata as an int32 tensor with the same bits (torch has no uint32 math)."""
    return torch.from_numpy(np.ascontiguousarray(words).view(np.int32))


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    if t is None:
        return None
    if not t.is_contiguous():
        raise ValueError("tensors must be contiguous")
    return t.data_ptr()


@dataclass
class Seq:
    """One sequence of a call (``starkv_seq``).  Tensor layouts as in starkv.h."""

    k: Optional[torch.Tensor] = None
    v: Optional[torch.Tensor] = None
    q: Optional[torch.Tensor] = None
    meta: Optional[torch.Tensor] = None     # int32 view of the u32 words
    meta_layer_stride: int = 0
    L: int = 0
    cur_frame: int = 0
    budget: int = 0
    slot: int = 0
    k_out: Optional[torch.Tensor] = None
    v_out: Optional[torch.Tensor] = None
    meta_out: Optional[torch.Tensor] = None
    idx: Optional[torch.Tensor] = None
    S: Optional[torch.Tensor] = None
    score: Optional[torch.Tensor] = None
    stats: Optional[torch.Tensor] = None
    meta_group_stride: int = 0              # per-KV-head mode: one metadata row per group
    lse: Optional[torch.Tensor] = None      # f32 [n_layers][H][w] supplied row normalisers
    attn_o: Optional[torch.Tensor] = None   # f32 [n_layers][H][w][d] window_attention output
    attn_lse: Optional[torch.Tensor] = None  # f32 [n_layers][H][w] window_attention normalisers

    def to_c(self) -> CSeq:
        s = CSeq()
        for name in ("k", "v", "q", "meta", "k_out", "v_out", "meta_out", "idx", "S", "score", "stats", "lse",
                     "attn_o", "attn_lse"):
            setattr(s, name, _ptr(getattr(self, name)))
        s.meta_layer_stride = self.meta_layer_stride
        s.meta_group_stride = self.meta_group_stride
        s.L, s.cur_frame, s.budget, s.slot = self.L, self.cur_frame, self.budget, self.slot
        return s


def _seq_array(seqs: Sequence[Seq]):
    arr = (CSeq * max(1, len(seqs)))()
    for i, s in enumerate(seqs):
        arr[i] = s.to_c()
    return arr


def _stream(stream) -> int:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream if torch.cuda.is_available() else 0
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


class State:
    """Owns a ``starkv_state`` (device-resident per-(slot, layer) state)."""

    def __init__(self, cfg: Config, stream=None):
        self.cfg = cfg
        self._c = cfg.to_c()
        h = C.c_void_p()
        _check(lib().starkv_init_state(C.byref(self._c), C.byref(h), _stream(stream)))
        self.handle = h

    def close(self) -> None:
        if self.handle:
            _check(lib().starkv_destroy_state(self.handle))
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def init_state(cfg: Config, stream=None) -> State:
    return State(cfg, stream)


def destroy_state(st: State) -> None:
    st.close()


def reset_seq(st: State, slot: int, stream=None) -> None:
    _check(lib().starkv_reset_seq(st.handle, slot, _stream(stream)))


def set_wait_limit(st: State, limit_ns: int) -> None:
    _check(lib().starkv_set_wait_limit(st.handle, int(limit_ns)))


def slot_state_bytes(st: State) -> int:
    n = C.c_size_t(0)
    _check(lib().starkv_slot_state_bytes(st.handle, C.byref(n)))
    return int(n.value)


def export_slot(st: State, slot: int, out: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """Slot ``slot``'s carried state (n, MI EMA, m_g of every layer) as a uint8
    host tensor (page-locked unless ``out`` is given); valid once the stream
    has been synchronised."""
    n = slot_state_bytes(st)
    if out is None:
        out = torch.empty(n, dtype=torch.uint8, pin_memory=torch.cuda.is_available())
    _check(lib().starkv_export_slot(st.handle, int(slot), out.data_ptr(), out.numel() * out.element_size(),
                                    _stream(stream)))
    return out


def import_slot(st: State, slot: int, buf: torch.Tensor, stream=None) -> None:
    """Replaces slot ``slot``'s carried state with one written by ``export_slot``."""
    _check(lib().starkv_import_slot(st.handle, int(slot), buf.data_ptr(), buf.numel() * buf.element_size(),
                                    _stream(stream)))


def selftest_wait(st: State, limit_ns: int, stream=None) -> None:
    """Runs the bounded-wait failure path once: a device wait that nothing
    completes gives up after ``limit_ns`` and latches ERR_TIMEOUT, which the
    next ``check_device_error`` raises."""
    _check(lib().starkv_selftest_wait(st.handle, int(limit_ns), _stream(stream)))


def workspace_bytes(st: State, seqs: Sequence[Seq], host: bool = False) -> int:
    arr = _seq_array(seqs)
    n = C.c_size_t()
    _check(lib().starkv_workspace_bytes(st.handle, arr, len(seqs), int(host), C.byref(n)))
    return int(n.value)


def workspace(st: State, seqs: Sequence[Seq], host: bool = False, device=None) -> torch.Tensor:
    return torch.empty(workspace_bytes(st, seqs, host), dtype=torch.uint8,
                       device=device or torch.device("cuda"))


def _call_layer(fn, st: State, layer: int, seqs: Sequence[Seq], ws: torch.Tensor, stream) -> None:
    arr = _seq_array(seqs)
    _check(fn(st.handle, layer, arr, len(seqs), ws.data_ptr(), ws.numel(), _stream(stream)))


def score_layer(st: State, layer: int, seqs: Sequence[Seq], ws: torch.Tensor, stream=None) -> None:
    _call_layer(lib().starkv_score_layer, st, layer, seqs, ws, stream)


def score_layer_noalloc(st: State, layer: int, seqs: Sequence[Seq], stream=None) -> None:
    """``starkv_score_layer`` without a workspace: for callers that cannot
    allocate device memory; the library's static 16 MiB scratch is used."""
    arr = _seq_array(seqs)
    _check(lib().starkv_score_layer_noalloc(st.handle, layer, arr, len(seqs), _stream(stream)))


def select(st: State, layer: int, seqs: Sequence[Seq], ws: torch.Tensor, stream=None) -> None:
    _call_layer(lib().starkv_select, st, layer, seqs, ws, stream)


def compact(st: State, layer: int, seqs: Sequence[Seq], ws: torch.Tensor, stream=None) -> None:
    _call_layer(lib().starkv_compact, st, layer, seqs, ws, stream)


def step(st: State, seqs: Sequence[Seq], ws: torch.Tensor, stream=None) -> None:
    arr = _seq_array(seqs)
    _check(lib().starkv_step(st.handle, arr, len(seqs), ws.data_ptr(), ws.numel(), _stream(stream)))


def window_attention(st: State, seqs: Sequence[Seq], ws: torch.Tensor, stream=None) -> None:
    """Attention output (``attn_o``, optional) and normaliser (``attn_lse``) of
    the window rows over the past keys, for every layer of every sequence."""
    arr = _seq_array(seqs)
    _check(lib().starkv_window_attention(st.handle, arr, len(seqs), ws.data_ptr(), ws.numel(),
                                         _stream(stream)))


def step_host(st: State, seqs: Sequence[Seq], ws: torch.Tensor, stream=None) -> None:
    arr = _seq_array(seqs)
    _check(lib().starkv_step_host(st.handle, arr, len(seqs), ws.data_ptr(), ws.numel(),
                                  _stream(stream)))


def check_device_error(st: State, stream=None) -> None:
    _check(lib().starkv_check_device_error(st.handle, _stream(stream)))


def device_error_status(st: State, stream=None) -> int:
    return lib().starkv_check_device_error(st.handle, _stream(stream))


def set_timing(st: State, on: bool) -> None:
    _check(lib().starkv_set_timing(st.handle, int(on)))


def kernel_times(st: State):
    """{kernel: (launches, total_ms)} since the previous read."""
    n = len(KERNELS)
    launches = (C.c_int64 * n)()
    ms = (C.c_float * n)()
    _check(lib().starkv_kernel_times(st.handle, launches, ms))
    return {k: (int(launches[i]), float(ms[i])) for i, k in enumerate(KERNELS)}
