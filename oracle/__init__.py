"""CPU oracle of the UltraMem memory-layer forward -- TEST INFRASTRUCTURE ONLY.

Loads ``ultramem_oracle.c`` (plain fp64 C, OpenMP over tokens) through ctypes.
Only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package; the product path never does.

Arrays are numpy: fp32 tensors as ``float32``, bf16 tensors as their raw
``uint16`` bit patterns, the Tucker cores and (u, t) as ``float32``.  The
paper's notation is kept: ``x, w_q, w_q_col, k_row, k_col, core, u, t, values,
w_proj, perm`` (see ``ultramem_oracle.h`` for shapes and equations).
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "ultramem_oracle.c")
_LIB_PATH = os.path.join(_HERE, "_ultramem_oracle.so")
_lock = threading.Lock()
_lib = None

F32, BF16 = 0, 1
ACT_NONE, ACT_SOFTMAX = 0, 1
SCORE_TUCKER, SCORE_PKM = 0, 1


class Config(C.Structure):
    _fields_ = [(name, C.c_int32) for name in (
        "d_in", "d_k", "heads", "rank", "n", "expand_e", "d_v", "d_out",
        "topk", "topm", "has_proj", "share_query", "act", "dtype", "cores", "conv_k",
        "query_ln", "score_mode")] + [("shuffle_seed", C.c_uint64), ("ln_eps", C.c_double)]


class Tensors(C.Structure):
    _fields_ = [("x", C.c_void_p), ("w_q", C.c_void_p), ("w_q_col", C.c_void_p),
                ("k_row", C.c_void_p), ("k_col", C.c_void_p),
                ("core", C.c_void_p), ("u", C.c_void_p), ("t", C.c_void_p),
                ("values", C.c_void_p), ("w_proj", C.c_void_p), ("perm", C.c_void_p),
                ("conv_w", C.c_void_p), ("conv_b", C.c_void_p), ("conv_state", C.c_void_p),
                ("seq_len", C.c_int64), ("ln_g", C.c_void_p), ("ln_b", C.c_void_p)]


def build(force: bool = False) -> str:
    """Compile the oracle shared library in place (gcc, -O2, OpenMP)."""
    if force or not os.path.exists(_LIB_PATH) or \
            os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + ".%d.tmp" % os.getpid()
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared",
                               "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = C.CDLL(build())
            P = C.c_void_p
            lib.uo_forward.argtypes = [P, P, C.c_int64, P, C.c_int64, P, P, P, C.c_int32]
            lib.uo_lookup_reduce.argtypes = [P, P, C.c_int64, P, P, P, C.c_int32]
            lib.uo_row_col_scores.argtypes = [P, P, C.c_int64, C.c_int64, C.c_int32, P, P]
            lib.uo_conv_state.argtypes = [P, P, C.c_int64, P]
            lib.uo_exact_topm.argtypes = [P, P, C.c_int64, P, C.c_int64, P, P, C.c_int32]
            lib.uo_lookup_reduce_backward.argtypes = [P, P, C.c_int64, P, P, P, P, P, P]
            lib.uo_key_ln.argtypes = [P, C.c_int32, C.c_int64, C.c_int32, P, P, C.c_double, P]
            lib.uo_rank1.argtypes = [P, C.c_int32, P, P, P]
            lib.uo_shuffle.argtypes = [P, P, C.c_int64]
            lib.uo_shuffle.restype = C.c_int64
            lib.uo_shuffle_params.argtypes = [C.c_uint64, C.c_uint64, P, P]
            lib.uo_splitmix64.argtypes = [C.c_uint64]
            lib.uo_splitmix64.restype = C.c_uint64
            _lib = lib
    return _lib


_CFG_KEYS = ("d_in", "d_k", "heads", "rank", "n", "expand_e", "d_v", "d_out", "topk",
             "topm", "has_proj", "share_query", "act", "dtype", "shuffle_seed")


def make_config(cfg: dict) -> Config:
    c = Config()
    for k in _CFG_KEYS:
        setattr(c, k, int(cfg[k]))
    c.cores = int(cfg.get("cores", 0))
    c.conv_k = int(cfg.get("conv_k", 0))
    c.query_ln = int(cfg.get("query_ln", 0))
    c.ln_eps = float(cfg.get("ln_eps", 1e-5))
    c.score_mode = int(cfg.get("score_mode", 0))
    return c


def cores_of(cfg: dict) -> int:
    """h, the component cores per head (Multi-Core Scoring, Sec. 3.2)."""
    return max(1, int(cfg.get("cores", 0)))


def keys_per_axis(cfg: dict) -> int:
    s = int(round(cfg["expand_e"] ** 0.5))
    return s * int(cfg["n"])


def _ptr(a):
    return None if a is None else a.ctypes.data


def _stored(a, dtype):
    """Checks that a stored tensor has the storage type the config names."""
    if a is None:
        return None
    want = np.uint16 if dtype == BF16 else np.float32
    if a.dtype != want:
        raise TypeError(f"oracle expects {want.__name__} storage, got {a.dtype}")
    return np.ascontiguousarray(a)


def _tensors(cfg: dict, t: dict):
    dt = int(cfg["dtype"])
    keep = {}
    for k in ("x", "w_q", "w_q_col", "k_row", "k_col", "values", "w_proj"):
        keep[k] = _stored(t.get(k), dt)
    for k in ("core", "u", "t", "conv_w", "conv_b", "ln_g", "ln_b"):
        a = t.get(k)
        keep[k] = None if a is None else np.ascontiguousarray(a, dtype=np.float32)
    keep["conv_state"] = _stored(t.get("conv_state"), dt)
    p = t.get("perm")
    keep["perm"] = None if p is None else np.ascontiguousarray(p, dtype=np.int64)
    s = Tensors(*[_ptr(keep[k]) for k in ("x", "w_q", "w_q_col", "k_row", "k_col",
                                          "core", "u", "t", "values", "w_proj", "perm",
                                          "conv_w", "conv_b", "conv_state")])
    s.seq_len = int(t.get("seq_len", 0))
    s.ln_g = _ptr(keep["ln_g"])
    s.ln_b = _ptr(keep["ln_b"])
    return s, keep


def forward(cfg: dict, tensors: dict, B: int, tokens=None, threads: int = 0):
    """Eq. 4-10 then Eq. 13-15 for the listed tokens (all B if None).

    Returns ``(out [n, d_out] f64, idx [n, H, m] i64, w [n, H, m] f64)``;
    with h > 1 component cores (MCS) ``w`` is ``[n, H, m, h]``, the score of
    each core at the slot."""
    lib = _load()
    c = make_config(cfg)
    s, keep = _tensors(cfg, tensors)
    tok = None if tokens is None else np.ascontiguousarray(tokens, dtype=np.int64)
    n = B if tok is None else len(tok)
    H, m = int(cfg["heads"]), int(cfg["topm"])
    out = np.zeros((n, int(cfg["d_out"])), np.float64)
    idx = np.zeros((n, H, m), np.int64)
    h = cores_of(cfg)
    w = np.zeros((n, H, m) if h == 1 else (n, H, m, h), np.float64)
    st = lib.uo_forward(C.byref(c), C.byref(s), int(B), _ptr(tok), int(n),
                        out.ctypes.data, idx.ctypes.data, w.ctypes.data, int(threads))
    del keep
    if st != 0:
        raise ValueError(f"uo_forward failed with status {st}")
    return out, idx, w


def exact_topm(cfg: dict, tensors: dict, B: int, tokens=None, threads: int = 0):
    """Eq. 5 (or Eq. 2 with PKM scoring) by brute force over the whole K x K
    grid: ``(idx [n, H, m] i64, w [n, H, m] f64)`` in uo_forward's order."""
    lib = _load()
    c = make_config(cfg)
    s, keep = _tensors(cfg, tensors)
    tok = None if tokens is None else np.ascontiguousarray(tokens, dtype=np.int64)
    n = B if tok is None else len(tok)
    H, m = int(cfg["heads"]), int(cfg["topm"])
    idx = np.zeros((n, H, m), np.int64)
    w = np.zeros((n, H, m), np.float64)
    st = lib.uo_exact_topm(C.byref(c), C.byref(s), int(B), _ptr(tok), int(n), idx.ctypes.data,
                           w.ctypes.data, int(threads))
    del keep
    if st != 0:
        raise ValueError(f"uo_exact_topm failed with status {st}")
    return idx, w


def lookup_reduce(cfg: dict, tensors: dict, idx, w, threads: int = 0):
    """Eq. 14-15 alone on given virtual addresses [n, H, m] and weights
    [n, H, m] (or [n, H, m, h], one per value slice, with h > 1 cores)."""
    lib = _load()
    c = make_config(cfg)
    s, keep = _tensors(cfg, tensors)
    idx = np.ascontiguousarray(idx, dtype=np.int64)
    w = np.ascontiguousarray(w, dtype=np.float64)
    n = idx.shape[0]
    if w.size != idx.size * cores_of(cfg):
        raise ValueError(f"weights {w.shape} do not match addresses {idx.shape}")
    out = np.zeros((n, int(cfg["d_out"])), np.float64)
    st = lib.uo_lookup_reduce(C.byref(c), C.byref(s), int(n), idx.ctypes.data,
                              w.ctypes.data, out.ctypes.data, int(threads))
    del keep
    if st != 0:
        raise ValueError(f"uo_lookup_reduce failed with status {st}")
    return out


def lookup_reduce_backward(cfg: dict, tensors: dict, idx, w, g):
    """Backward of Eq. 14-15 for slots idx [n, H, m], weights w [n, H, m]
    (or [n, H, m, h]) and dL/do g [n, d_out] (stored type): ``(dv [N, d_v],
    dw (w's shape), dwp [E, d_v, d_out])`` in f64, dv accumulated from 0."""
    lib = _load()
    c = make_config(cfg)
    s, keep = _tensors(cfg, tensors)
    idx = np.ascontiguousarray(idx, dtype=np.int64)
    w = np.ascontiguousarray(w, dtype=np.float64)
    g = _stored(np.asarray(g), int(cfg["dtype"]))
    n = idx.shape[0]
    N = int(cfg["n"]) ** 2
    E, dv_, do = int(cfg["expand_e"]), int(cfg["d_v"]), int(cfg["d_out"])
    dv = np.zeros((N, dv_), np.float64)
    dw = np.zeros(w.shape, np.float64)
    dwp = np.zeros((E, dv_, do), np.float64)
    st = lib.uo_lookup_reduce_backward(C.byref(c), C.byref(s), int(n), idx.ctypes.data,
                                       w.ctypes.data, g.ctypes.data, dv.ctypes.data,
                                       dw.ctypes.data, dwp.ctypes.data)
    del keep
    if st != 0:
        raise ValueError(f"uo_lookup_reduce_backward failed with status {st}")
    return dv, dw, dwp


def row_col_scores(cfg: dict, tensors: dict, b: int, h: int, B: int | None = None):
    """Eq. 4 for token b of the batch (B tokens, default all rows of x),
    head h: ``(S_row [r, K], S_col [r, K])`` in fp64."""
    lib = _load()
    c = make_config(cfg)
    s, keep = _tensors(cfg, tensors)
    r, K = int(cfg["rank"]), keys_per_axis(cfg)
    if B is None:
        B = np.asarray(tensors["x"]).shape[0]
    sr = np.zeros((r, K), np.float64)
    sc = np.zeros((r, K), np.float64)
    st = lib.uo_row_col_scores(C.byref(c), C.byref(s), int(B), int(b), int(h),
                               sr.ctypes.data, sc.ctypes.data)
    del keep
    if st != 0:
        raise ValueError(f"uo_row_col_scores failed with status {st}")
    return sr, sc


def conv_state(cfg: dict, tensors: dict, B: int):
    """Trick 4's state after a batch of B tokens: [B/seq_len, conv_k-1, d_in]
    f64, the last conv_k - 1 inputs of each sequence, oldest first."""
    lib = _load()
    c = make_config(cfg)
    s, keep = _tensors(cfg, tensors)
    L = int(tensors.get("seq_len", 0)) or B
    out = np.zeros((B // L, int(cfg["conv_k"]) - 1, int(cfg["d_in"])), np.float64)
    st = lib.uo_conv_state(C.byref(c), C.byref(s), int(B), out.ctypes.data)
    del keep
    if st != 0:
        raise ValueError(f"uo_conv_state failed with status {st}")
    return out


def key_ln(keys, dtype: int, g, b=None, eps: float = 1e-5):
    """Trick 2 for keys: LayerNorm of each row of ``keys`` [..., d] (stored
    as ``dtype``) with gain g [d] and bias b [d]; f64 of the same shape."""
    lib = _load()
    k = _stored(np.asarray(keys), dtype)
    g = np.ascontiguousarray(g, dtype=np.float32)
    bb = None if b is None else np.ascontiguousarray(b, dtype=np.float32)
    d = k.shape[-1]
    out = np.zeros(k.shape, np.float64)
    st = lib.uo_key_ln(k.ctypes.data, int(dtype), int(k.size // d), int(d), g.ctypes.data,
                       _ptr(bb), float(eps), out.ctypes.data)
    if st != 0:
        raise ValueError(f"uo_key_ln failed with status {st}")
    return out


def rank1(core):
    """Leading singular triplet ``(u, t, sigma)`` of one r x r core (Eq. 7)."""
    lib = _load()
    c = np.ascontiguousarray(core, dtype=np.float64)
    r = c.shape[0]
    u = np.zeros(r, np.float64)
    t = np.zeros(r, np.float64)
    sig = np.zeros(1, np.float64)
    st = lib.uo_rank1(c.ctypes.data, r, u.ctypes.data, t.ctypes.data, sig.ctypes.data)
    if st != 0:
        raise ValueError(f"uo_rank1 failed with status {st}")
    return u, t, float(sig[0])


def shuffle(cfg: dict, v, perm=None):
    """Eq. 14: shuffled virtual addresses for an array of addresses."""
    lib = _load()
    c = make_config(cfg)
    p = None if perm is None else np.ascontiguousarray(perm, dtype=np.int64)
    v = np.asarray(v, dtype=np.int64)
    out = np.array([lib.uo_shuffle(C.byref(c), _ptr(p), int(e)) for e in v.ravel()],
                   dtype=np.int64)
    return out.reshape(v.shape)


def shuffle_params(seed: int, m: int):
    lib = _load()
    a = C.c_uint64()
    c = C.c_uint64()
    lib.uo_shuffle_params(C.c_uint64(seed), C.c_uint64(m), C.byref(a), C.byref(c))
    return a.value, c.value


def splitmix64(state: int) -> int:
    """First output of a SplitMix64 generator in the given state."""
    return int(_load().uo_splitmix64(C.c_uint64(state)))
