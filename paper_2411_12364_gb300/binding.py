"""Thin Python binding of libultramem.so (include/ultramem.h).

Argument marshalling only: torch tensors become device pointers and the
current torch stream becomes the cudaStream_t; every step of the layer runs
in the CUDA library.  There is no fallback: if the library cannot be built or
loaded, or no GPU is present, the calls raise.
"""
from __future__ import annotations

import ctypes as C
import os
import threading

import torch

from . import build as _build

OK, EINVAL, ENOMEM, ECUDA, ETIMEOUT, EDEVICE, ENODEV = 0, -1, -2, -3, -4, -5, -6
F32, BF16 = 0, 1
ACT_NONE, ACT_SOFTMAX = 0, 1
SCORE_TUCKER, SCORE_PKM = 0, 1

# every function include/ultramem.h declares
EXPORTS = ("ultramem_create", "ultramem_destroy", "ultramem_forward",
           "ultramem_forward_host", "ultramem_retrieve", "ultramem_lookup_reduce",
           "ultramem_check", "ultramem_rank1", "ultramem_profile_enable",
           "ultramem_profile_read", "ultramem_stage_name", "ultramem_status_string",
           "ultramem_last_error", "ultramem_version", "ultramem_lookup_reduce_noalloc",
           "ultramem_last_launches", "ultramem_forward_seq", "ultramem_key_ln",
           "ultramem_retrieve_exact", "ultramem_lookup_reduce_backward",
           "ultramem_debug_wait_probe", "ultramem_debug_fail_alloc",
           "ultramem_debug_live_allocations", "ultramem_debug_candidates",
           "ultramem_shard_route", "ultramem_shard_lookup", "ultramem_shard_pool")


class Config(C.Structure):
    _fields_ = [(name, C.c_int32) for name in (
        "d_in", "d_k", "heads", "rank", "n", "expand_e", "d_v", "d_out", "topk", "topm",
        "has_proj", "share_query", "act", "dtype", "max_tokens", "cores", "conv_k",
        "query_ln", "score_mode")] + [("shuffle_seed", C.c_uint64), ("ln_eps", C.c_float),
                                     ("shard_rows", C.c_int64)]


class Weights(C.Structure):
    _fields_ = [("w_q", C.c_void_p), ("w_q_col", C.c_void_p), ("k_row", C.c_void_p),
                ("k_col", C.c_void_p), ("core", C.c_void_p), ("u", C.c_void_p),
                ("t", C.c_void_p), ("values", C.c_void_p), ("w_proj", C.c_void_p),
                ("perm", C.c_void_p), ("conv_w", C.c_void_p), ("conv_b", C.c_void_p),
                ("ln_g", C.c_void_p), ("ln_b", C.c_void_p)]


class UltraMemError(RuntimeError):
    def __init__(self, status: int, what: str):
        msg = f"{what}: {status_string(status)} ({status})"
        if status in (ECUDA, ENOMEM):
            detail = load().ultramem_last_error().decode()
            if detail:
                msg += f" [{detail}]"
        super().__init__(msg)
        self.status = status


_lib = None
_lock = threading.Lock()


def load(path: str | None = None) -> C.CDLL:
    """Builds (if needed) and loads the CUDA library."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        path = path or _build.build()
        lib = C.CDLL(path)
        P, I32, I64 = C.c_void_p, C.c_int32, C.c_int64
        lib.ultramem_create.argtypes = [P, P, P]
        lib.ultramem_create.restype = I32
        lib.ultramem_destroy.argtypes = [P]
        lib.ultramem_destroy.restype = None
        lib.ultramem_forward.argtypes = [P, P, I32, P, P, P, P]
        lib.ultramem_forward.restype = I32
        lib.ultramem_forward_seq.argtypes = [P, P, I32, I32, P, P, P, P, P, P]
        lib.ultramem_forward_seq.restype = I32
        lib.ultramem_key_ln.argtypes = [P, I32, I64, I32, P, P, C.c_float, P, P]
        lib.ultramem_key_ln.restype = I32
        lib.ultramem_forward_host.argtypes = [P, P, I32, P, P]
        lib.ultramem_forward_host.restype = I32
        lib.ultramem_retrieve.argtypes = [P, P, I32, P, P, P]
        lib.ultramem_retrieve_exact.argtypes = [P, P, I32, P, P, P]
        lib.ultramem_retrieve_exact.restype = I32
        lib.ultramem_lookup_reduce_backward.argtypes = [P, P, P, P, I32, P, P, P, P]
        lib.ultramem_lookup_reduce_backward.restype = I32
        lib.ultramem_retrieve.restype = I32
        lib.ultramem_lookup_reduce.argtypes = [P, P, P, I32, P, P]
        lib.ultramem_lookup_reduce.restype = I32
        lib.ultramem_check.argtypes = [P, P]
        lib.ultramem_check.restype = I32
        lib.ultramem_rank1.argtypes = [P, I32, P, P, P]
        lib.ultramem_rank1.restype = I32
        lib.ultramem_profile_enable.argtypes = [P, I32]
        lib.ultramem_profile_enable.restype = I32
        lib.ultramem_profile_read.argtypes = [P, P, I32]
        lib.ultramem_profile_read.restype = I32
        lib.ultramem_stage_name.argtypes = [I32]
        lib.ultramem_stage_name.restype = C.c_char_p
        lib.ultramem_status_string.argtypes = [I32]
        lib.ultramem_status_string.restype = C.c_char_p
        lib.ultramem_lookup_reduce_noalloc.argtypes = [P, P, P, P, P, P, I32, P, P]
        lib.ultramem_lookup_reduce_noalloc.restype = I32
        lib.ultramem_last_launches.argtypes = [P]
        lib.ultramem_last_launches.restype = I32
        lib.ultramem_last_error.argtypes = []
        lib.ultramem_last_error.restype = C.c_char_p
        lib.ultramem_version.argtypes = []
        lib.ultramem_version.restype = I32
        lib.ultramem_debug_wait_probe.argtypes = [P]
        lib.ultramem_debug_wait_probe.restype = I32
        lib.ultramem_debug_fail_alloc.argtypes = [I32]
        lib.ultramem_debug_fail_alloc.restype = None
        lib.ultramem_debug_live_allocations.argtypes = []
        lib.ultramem_debug_live_allocations.restype = I32
        lib.ultramem_debug_candidates.argtypes = [P, I32]
        lib.ultramem_debug_candidates.restype = I32
        lib.ultramem_shard_route.argtypes = [P, P, I32, I32, I64, P, P, P, P]
        lib.ultramem_shard_route.restype = I32
        lib.ultramem_shard_lookup.argtypes = [P, P, I64, P, P]
        lib.ultramem_shard_lookup.restype = I32
        lib.ultramem_shard_pool.argtypes = [P, P, P, I32, P, P, P, P]
        lib.ultramem_shard_pool.restype = I32
        _lib = lib
        return lib


def status_string(s: int) -> str:
    return load().ultramem_status_string(int(s)).decode()


def _check(status: int, what: str):
    if status != OK:
        raise UltraMemError(status, what)


def rank1(core):
    """Leading singular triplet (u, t, sigma) of one r x r core, Eq. 7."""
    import numpy as np
    c = np.ascontiguousarray(core, dtype=np.float32)
    r = c.shape[0]
    u = np.zeros(r, np.float32)
    t = np.zeros(r, np.float32)
    s = np.zeros(1, np.float32)
    _check(load().ultramem_rank1(c.ctypes.data, r, u.ctypes.data, t.ctypes.data,
                                 s.ctypes.data), "ultramem_rank1")
    return u, t, float(s[0])


def _ptr(t):
    return None if t is None else t.data_ptr()


def key_ln(keys: torch.Tensor, g: torch.Tensor, b: torch.Tensor | None = None,
           eps: float = 1e-5, out: torch.Tensor | None = None) -> torch.Tensor:
    """Trick 2 for keys: LayerNorm of each row of ``keys`` (fp32 or bf16 on
    the device) with gain g and bias b (fp32), in the keys' type."""
    lib = load()
    keys = keys.contiguous()
    dt = {torch.float32: F32, torch.bfloat16: BF16}[keys.dtype]
    d = keys.shape[-1]
    out = torch.empty_like(keys) if out is None else out
    g = g.to(torch.float32).contiguous()
    bb = None if b is None else b.to(torch.float32).contiguous()
    _check(lib.ultramem_key_ln(keys.data_ptr(), dt, keys.numel() // d, d, g.data_ptr(),
                               _ptr(bb), float(eps), out.data_ptr(), _stream()),
           "ultramem_key_ln")
    return out


# The raw handle of the current stream without building a torch.cuda.Stream
# object (which costs about 3 us a call, a tenth of a decode step).
_raw_stream = getattr(torch._C, "_cuda_getCurrentRawStream", None)


def _stream():
    if _raw_stream is not None:
        return _raw_stream(torch.cuda.current_device())
    return torch.cuda.current_stream().cuda_stream


_CFG_KEYS = ("d_in", "d_k", "heads", "rank", "n", "expand_e", "d_v", "d_out", "topk",
             "topm", "has_proj", "share_query", "act", "dtype")


class UltraMemLayer:
    """One UltraMem layer on the current CUDA device.

    ``weights`` holds device tensors in the layer's storage type (``w_q``,
    ``w_q_col``, ``k_row``, ``k_col``, ``values``, ``w_proj``), the cores
    ``core`` [H, r, r] (with ``cfg["cores"]`` = h > 1 component cores,
    [H, h, r, r]; any device, fp32) and optionally ``u``, ``t`` [H, r] and an
    explicit shuffle ``perm`` (int32/uint32 device tensor).  The layer keeps
    references to them for its lifetime.  Slot weights ``w`` are [B, H, m],
    or [B, H, m, h] with h > 1 cores (one per value slice, Eq. 17)."""

    def __init__(self, cfg: dict, weights: dict, max_tokens: int):
        if not torch.cuda.is_available():
            raise RuntimeError("UltraMemLayer needs a CUDA device (GB300, sm_103a)")
        self.lib = load()
        self.cfg = dict(cfg)
        c = Config()
        for k in _CFG_KEYS:
            setattr(c, k, int(cfg[k]))
        c.max_tokens = int(max_tokens)
        c.cores = int(cfg.get("cores", 0))
        c.conv_k = int(cfg.get("conv_k", 0))
        c.query_ln = int(cfg.get("query_ln", 0))
        c.ln_eps = float(cfg.get("ln_eps", 1e-5))
        c.score_mode = int(cfg.get("score_mode", 0))
        c.shuffle_seed = int(cfg.get("shuffle_seed", 0))
        c.shard_rows = int(cfg.get("shard_rows", 0))
        self._c = c
        dev_keys = ("w_q", "w_q_col", "k_row", "k_col", "values", "w_proj", "perm", "conv_w",
                    "conv_b", "ln_g", "ln_b")
        self._keep = {k: (None if weights.get(k) is None else weights[k].contiguous())
                      for k in dev_keys}
        for k, v in self._keep.items():
            if v is not None and not v.is_cuda:
                raise ValueError(f"{k} must be a CUDA tensor")
        core = weights.get("core")
        self._core = None if core is None else \
            core.detach().to("cpu", torch.float32).contiguous()
        u, t = weights.get("u"), weights.get("t")
        self._u = None if u is None else torch.as_tensor(u).to("cpu", torch.float32).contiguous()
        self._t = None if t is None else torch.as_tensor(t).to("cpu", torch.float32).contiguous()
        w = Weights(_ptr(self._keep["w_q"]), _ptr(self._keep["w_q_col"]),
                    _ptr(self._keep["k_row"]), _ptr(self._keep["k_col"]),
                    _ptr(self._core), _ptr(self._u), _ptr(self._t),
                    _ptr(self._keep["values"]), _ptr(self._keep["w_proj"]),
                    _ptr(self._keep["perm"]), _ptr(self._keep["conv_w"]),
                    _ptr(self._keep["conv_b"]), _ptr(self._keep["ln_g"]),
                    _ptr(self._keep["ln_b"]))
        h = C.c_void_p()
        _check(self.lib.ultramem_create(C.byref(c), C.byref(w), C.byref(h)), "ultramem_create")
        self._h = h
        self.max_tokens = int(max_tokens)
        self.dtype = torch.float32 if int(cfg["dtype"]) == F32 else torch.bfloat16
        self.cores = max(1, int(cfg.get("cores", 0)))

    def _w_shape(self, B: int):
        H, m = int(self.cfg["heads"]), int(self.cfg["topm"])
        return (B, H, m) if self.cores == 1 else (B, H, m, self.cores)

    # -- calls ------------------------------------------------------------
    def forward(self, x: torch.Tensor, out: torch.Tensor | None = None, with_slots=False):
        """S1-S9.  Returns out [B, D'_v] (and idx [B,H,m] int64, w [B,H,m] fp32
        when ``with_slots``)."""
        x = x.contiguous()
        B = x.shape[0]
        if out is None:
            out = torch.empty((B, int(self.cfg["d_out"])), dtype=self.dtype, device=x.device)
        idx = w = None
        if with_slots:
            H, m = int(self.cfg["heads"]), int(self.cfg["topm"])
            idx = torch.empty((B, H, m), dtype=torch.int64, device=x.device)
            w = torch.empty(self._w_shape(B), dtype=torch.float32, device=x.device)
        _check(self.lib.ultramem_forward(self._h, x.data_ptr(), B, out.data_ptr(), _ptr(idx),
                                         _ptr(w), _stream()), "ultramem_forward")
        return (out, idx, w) if with_slots else out

    def forward_seq(self, x: torch.Tensor, n_seq: int, state_in=None, state_out=None,
                    out: torch.Tensor | None = None, with_slots=False):
        """S1-S9 on n_seq sequences back to back in x [n_seq*L, D_i]; the
        query convolution (Trick 4) reads state_in [n_seq, conv_k-1, D_i]
        before each sequence and writes state_out (both optional)."""
        x = x.contiguous()
        B = x.shape[0]
        if n_seq < 1 or B % n_seq:
            raise ValueError(f"{B} tokens do not split into {n_seq} sequences")
        if out is None:
            out = torch.empty((B, int(self.cfg["d_out"])), dtype=self.dtype, device=x.device)
        idx = w = None
        if with_slots:
            H, m = int(self.cfg["heads"]), int(self.cfg["topm"])
            idx = torch.empty((B, H, m), dtype=torch.int64, device=x.device)
            w = torch.empty(self._w_shape(B), dtype=torch.float32, device=x.device)
        si = None if state_in is None else state_in.contiguous()
        _check(self.lib.ultramem_forward_seq(self._h, x.data_ptr(), n_seq, B // n_seq, _ptr(si),
                                             _ptr(state_out), out.data_ptr(), _ptr(idx),
                                             _ptr(w), _stream()), "ultramem_forward_seq")
        return (out, idx, w) if with_slots else out

    def forward_host(self, x_host: torch.Tensor, out_host: torch.Tensor):
        """The forward on host tensors (pinned for asynchronous copies)."""
        _check(self.lib.ultramem_forward_host(self._h, x_host.data_ptr(), x_host.shape[0],
                                              out_host.data_ptr(), _stream()),
               "ultramem_forward_host")
        return out_host

    def retrieve(self, x: torch.Tensor):
        """S1-S6: (idx [B,H,m] int64 virtual addresses, w [B,H,m] fp32)."""
        x = x.contiguous()
        B = x.shape[0]
        H, m = int(self.cfg["heads"]), int(self.cfg["topm"])
        idx = torch.empty((B, H, m), dtype=torch.int64, device=x.device)
        w = torch.empty(self._w_shape(B), dtype=torch.float32, device=x.device)
        _check(self.lib.ultramem_retrieve(self._h, x.data_ptr(), B, idx.data_ptr(),
                                          w.data_ptr(), _stream()), "ultramem_retrieve")
        return idx, w

    def retrieve_exact(self, x: torch.Tensor):
        """Eq. 5 (Eq. 2 for product keys) by brute force over each head's
        whole grid: (idx [B,H,m] int64, w [B,H,m] fp32 raw scores)."""
        x = x.contiguous()
        B = x.shape[0]
        H, m = int(self.cfg["heads"]), int(self.cfg["topm"])
        idx = torch.empty((B, H, m), dtype=torch.int64, device=x.device)
        w = torch.empty((B, H, m), dtype=torch.float32, device=x.device)
        _check(self.lib.ultramem_retrieve_exact(self._h, x.data_ptr(), B, idx.data_ptr(),
                                                w.data_ptr(), _stream()),
               "ultramem_retrieve_exact")
        return idx, w

    def lookup_reduce(self, idx: torch.Tensor, w: torch.Tensor):
        """S7-S9 on given slots (Eq. 14-15)."""
        idx = idx.contiguous().to(torch.int64)
        w = w.contiguous().to(torch.float32)
        B = idx.shape[0]
        if w.numel() != idx.numel() * self.cores:
            raise ValueError(f"weights {tuple(w.shape)} do not match addresses {tuple(idx.shape)}")
        out = torch.empty((B, int(self.cfg["d_out"])), dtype=self.dtype, device=idx.device)
        _check(self.lib.ultramem_lookup_reduce(self._h, idx.data_ptr(), w.data_ptr(), B,
                                               out.data_ptr(), _stream()),
               "ultramem_lookup_reduce")
        return out

    def lookup_reduce_backward(self, idx: torch.Tensor, w: torch.Tensor, g: torch.Tensor,
                               dvalues: torch.Tensor | None = None, want_dw=True,
                               want_dw_proj=True):
        """Backward of S7-S9: (dvalues [N, D_v] fp32, accumulated into the given
        tensor or a new zero one; dw like w; dw_proj [E, D_v, D'_v] or None)."""
        idx = idx.contiguous().to(torch.int64)
        w = w.contiguous().to(torch.float32)
        g = g.contiguous().to(self.dtype)
        B = idx.shape[0]
        c = self.cfg
        N = int(c["n"]) ** 2
        if dvalues is None:
            dvalues = torch.zeros((N, int(c["d_v"])), dtype=torch.float32, device=idx.device)
        dw = torch.empty_like(w) if want_dw else None
        dwp = torch.empty((int(c["expand_e"]), int(c["d_v"]), int(c["d_out"])),
                          dtype=torch.float32, device=idx.device) \
            if want_dw_proj and int(c["has_proj"]) else None
        _check(self.lib.ultramem_lookup_reduce_backward(
            self._h, idx.data_ptr(), w.data_ptr(), g.data_ptr(), B, _ptr(dvalues), _ptr(dw),
            _ptr(dwp), _stream()), "ultramem_lookup_reduce_backward")
        return dvalues, dw, dwp

    # -- number-wise partitioned table (App. D) ---------------------------
    def shard_route(self, idx: torch.Tensor, P: int, rows_per_rank: int):
        """Slots idx [n,H,m] grouped by the rank that owns their row:
        (counts [P], send_rows [S], slot_pos [S]), int32 device tensors."""
        idx = idx.contiguous().to(torch.int64)
        S = idx.numel()
        counts = torch.empty(P, dtype=torch.int32, device=idx.device)
        send_rows = torch.empty(S, dtype=torch.int32, device=idx.device)
        slot_pos = torch.empty(S, dtype=torch.int32, device=idx.device)
        _check(self.lib.ultramem_shard_route(self._h, idx.data_ptr(), idx.shape[0], int(P),
                                             int(rows_per_rank), counts.data_ptr(),
                                             send_rows.data_ptr(), slot_pos.data_ptr(),
                                             _stream()), "ultramem_shard_route")
        return counts, send_rows, slot_pos

    def shard_lookup(self, rows: torch.Tensor):
        """Rows of this layer's table (its shard) at local indices ``rows``."""
        rows = rows.contiguous().to(torch.int32)
        out = torch.empty((rows.numel(), int(self.cfg["d_v"])), dtype=self.dtype,
                          device=rows.device)
        _check(self.lib.ultramem_shard_lookup(self._h, rows.data_ptr(), rows.numel(),
                                              out.data_ptr(), _stream()),
               "ultramem_shard_lookup")
        return out

    def shard_pool(self, idx: torch.Tensor, w: torch.Tensor, slot_pos: torch.Tensor,
                   back_rows: torch.Tensor):
        """Eq. 15 pooling and the projection on the rows the owners returned."""
        idx = idx.contiguous().to(torch.int64)
        w = w.contiguous().to(torch.float32)
        back_rows = back_rows.contiguous()
        out = torch.empty((idx.shape[0], int(self.cfg["d_out"])), dtype=self.dtype,
                          device=idx.device)
        _check(self.lib.ultramem_shard_pool(self._h, idx.data_ptr(), w.data_ptr(), idx.shape[0],
                                            slot_pos.contiguous().data_ptr(),
                                            back_rows.data_ptr(), out.data_ptr(), _stream()),
               "ultramem_shard_pool")
        return out

    def check(self) -> int:
        """Syncs the current stream and returns the device error status."""
        return int(self.lib.ultramem_check(self._h, _stream()))

    def candidates(self, mode: int):
        """Scoring form (test hook): 0 every key, 1 candidate lists, 2 lists on
        long grids only (the default)."""
        _check(self.lib.ultramem_debug_candidates(self._h, int(mode)), "debug_candidates")

    def last_launches(self) -> int:
        """Kernels launched by the most recent successful call on this layer."""
        return int(self.lib.ultramem_last_launches(self._h))

    def profile(self, enable: bool = True):
        _check(self.lib.ultramem_profile_enable(self._h, int(enable)), "profile_enable")

    def profile_read(self, gaps: bool = False):
        """Device time (ms) of each stage of the most recent profiled
        forward; with ``gaps`` also the hand-off before each stage."""
        buf = (C.c_float * 10)()
        n = self.lib.ultramem_profile_read(self._h, buf, 10)
        ns = min(n, 5)
        names = [self.lib.ultramem_stage_name(i).decode() for i in range(ns)]
        times = {names[i]: float(buf[i]) for i in range(ns)}
        if not gaps:
            return times
        return times, {names[i]: float(buf[5 + i]) for i in range(ns)} if n >= 10 else {}

    def close(self):
        if getattr(self, "_h", None):
            self.lib.ultramem_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
