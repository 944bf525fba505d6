"""The C-ABI library builds, loads and exports every symbol include/ultramem.h
declares; its host-only helpers behave (no GPU needed)."""
import ctypes as C
import os
import re

import numpy as np
import pytest

from paper_2411_12364_gb300 import binding

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))),
                      "include", "ultramem.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(ultramem_[a-z0-9_]+)\s*\(", text)))


def test_library_exports_every_declared_function():
    lib = binding.load()
    names = declared_functions()
    assert len(names) >= 13
    for n in names:
        assert hasattr(lib, n), f"{n} is declared but not exported"
    assert set(names) == set(binding.EXPORTS)


def test_version_and_status_strings():
    lib = binding.load()
    assert lib.ultramem_version() == 2
    for s in (0, -1, -2, -3, -4, -5, -6):
        assert binding.status_string(s) not in ("", "unknown status")
    assert binding.status_string(-99) == "unknown status"
    assert lib.ultramem_stage_name(0).decode() == "query"
    assert lib.ultramem_stage_name(99) is None


@pytest.mark.parametrize("r", [1, 2, 3, 5, 8])
def test_host_rank1_matches_numpy_svd(r):
    """The library's create-time SVD (one-sided Jacobi) against numpy."""
    rng = np.random.default_rng(r)
    for _ in range(10):
        Cm = rng.normal(size=(r, r)).astype(np.float32)
        u, t, s = binding.rank1(Cm)
        U, S, Vt = np.linalg.svd(Cm.astype(np.float64))
        assert abs(s - S[0]) < 1e-5 * S[0]
        assert u.sum() > 0
        np.testing.assert_allclose(Cm.astype(np.float64) @ t, s * u, atol=2e-5 * S[0])
        if S.size > 1 and S[0] - S[1] > 1e-3:
            sgn = np.sign(U[:, 0] @ u)
            np.testing.assert_allclose(u, sgn * U[:, 0], atol=1e-5)
            np.testing.assert_allclose(t, sgn * Vt[0], atol=1e-5)


def test_host_rank1_rejects_zero_core():
    with pytest.raises(binding.UltraMemError) as e:
        binding.rank1(np.zeros((2, 2), np.float32))
    assert e.value.status == binding.EINVAL


def _create(cfg_over=None, **w_over):
    lib = binding.load()
    c = binding.Config(d_in=64, d_k=32, heads=2, rank=2, n=16, expand_e=4, d_v=64, d_out=96,
                       topk=8, topm=8, has_proj=1, share_query=1, act=0, dtype=1,
                       max_tokens=16, cores=0, shuffle_seed=3)
    for k, v in (cfg_over or {}).items():
        setattr(c, k, v)
    core = np.ones((2, 2, 2), np.float32)
    fake = 4096  # never dereferenced: validation rejects before any device use
    w = binding.Weights(fake, None, fake, fake, core.ctypes.data, None, None, fake, fake, None)
    for k, v in w_over.items():
        setattr(w, k, v)
    h = C.c_void_p()
    st = lib.ultramem_create(C.byref(c), C.byref(w), C.byref(h))
    return st, h


@pytest.mark.parametrize("bad", [dict(rank=3), dict(expand_e=3), dict(expand_e=25),
                                 dict(topk=200), dict(topm=65), dict(d_v=60),
                                 dict(has_proj=0), dict(act=7), dict(dtype=9),
                                 dict(max_tokens=0), dict(n=30000),
                                 dict(rank=9, d_k=36), dict(cores=-1), dict(cores=9),
                                 dict(cores=2, act=1), dict(cores=3), dict(cores=16),
                                 dict(conv_k=2), dict(conv_k=-1), dict(query_ln=1),
                                 dict(query_ln=2), dict(score_mode=2), dict(score_mode=1),
                                 dict(heads=65), dict(d_k=8192),
                                 dict(score_mode=1, rank=1, d_k=32, cores=2)])
def test_create_rejects_invalid_configs(bad):
    st, h = _create(bad)
    assert st == binding.EINVAL
    assert not h.value


def test_create_rejects_missing_or_misaligned_tensors():
    assert _create(None, values=None)[0] == binding.EINVAL
    assert _create(None, values=4098)[0] == binding.EINVAL          # not 16-byte aligned
    assert _create(dict(share_query=0))[0] == binding.EINVAL         # no W_q_col
    assert _create(None, w_proj=None)[0] == binding.EINVAL
    u = np.ones(4, np.float32)
    assert _create(None, u=u.ctypes.data)[0] == binding.EINVAL       # u without t


def test_null_handle_calls_are_rejected():
    lib = binding.load()
    assert lib.ultramem_forward(None, None, 1, None, None, None, None) == binding.EINVAL
    assert lib.ultramem_lookup_reduce(None, None, None, 1, None, None) == binding.EINVAL
    assert lib.ultramem_check(None, None) == binding.EINVAL
    assert lib.ultramem_forward_seq(None, None, 1, 1, None, None, None, None, None,
                                    None) == binding.EINVAL
    assert lib.ultramem_retrieve_exact(None, None, 1, None, None, None) == binding.EINVAL
    assert lib.ultramem_lookup_reduce_backward(None, None, None, None, 1, None, None, None,
                                               None) == binding.EINVAL
    assert lib.ultramem_last_launches(None) == 0
    lib.ultramem_destroy(None)


def test_key_ln_rejects_invalid_arguments():
    """Checked before anything is launched (no device needed)."""
    lib = binding.load()
    fake = 4096   # never dereferenced
    assert lib.ultramem_key_ln(None, 1, 4, 8, fake, None, 1e-5, fake, None) == binding.EINVAL
    assert lib.ultramem_key_ln(fake, 7, 4, 8, fake, None, 1e-5, fake, None) == binding.EINVAL
    assert lib.ultramem_key_ln(fake, 1, 4, 0, fake, None, 1e-5, fake, None) == binding.EINVAL
    assert lib.ultramem_key_ln(fake, 1, -1, 8, fake, None, 1e-5, fake, None) == binding.EINVAL
    assert lib.ultramem_key_ln(fake, 1, 4, 8, fake, None, -1.0, fake, None) == binding.EINVAL
    assert lib.ultramem_key_ln(fake, 1, 4, 8, None, None, 1e-5, fake, None) == binding.EINVAL
