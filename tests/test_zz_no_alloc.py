"""ultramem_lookup_reduce_noalloc: the lookup-reduce for callers that cannot
allocate device memory (no layer handle, scratch in static device memory).
Its output must match the oracle's lookup-reduce (Eq. 14-15) and the
handle-based ultramem_lookup_reduce on the same slots, on two calls in a
row (the static scratch keeps the previous call's contents), also with an
explicit shuffle table and with addresses outside the grid (skipped, as a
slot of weight 0).  Collected last so that a failure here cannot hide the
others."""
import ctypes as C

import numpy as np
import pytest
import torch

import oracle
from paper_2411_12364_gb300 import binding, workloads
from tests import parity

pytestmark = pytest.mark.gpu


def _config_struct(cfg, max_tokens):
    c = binding.Config()
    for k in ("d_in", "d_k", "heads", "rank", "n", "expand_e", "d_v", "d_out", "topk", "topm",
              "has_proj", "share_query", "act", "dtype"):
        setattr(c, k, int(cfg[k]))
    c.max_tokens = max_tokens
    c.cores = int(cfg.get("cores", 0))
    c.shuffle_seed = int(cfg["shuffle_seed"])
    return c


def _noalloc(lib, c, w, idx, wt, out, perm=None):
    st = lib.ultramem_lookup_reduce_noalloc(
        C.byref(c), w["values"].data_ptr(),
        None if w.get("w_proj") is None else w["w_proj"].data_ptr(),
        None if perm is None else perm.data_ptr(),
        idx.data_ptr(), wt.data_ptr(), idx.shape[0], out.data_ptr(),
        torch.cuda.current_stream().cuda_stream)
    return st


def _oracle_out(cfg, w, idx, wt, perm=None):
    """The oracle's lookup-reduce of the given slots; an address outside
    [0, E N) contributes nothing (the kernels skip it)."""
    t = {k: workloads.stored_numpy(v) for k, v in w.items() if k in ("values", "w_proj")}
    if perm is not None:
        t["perm"] = perm.cpu().numpy().astype(np.int64)
    i = idx.cpu().numpy().copy()
    ww = wt.cpu().numpy().astype(np.float64).copy()
    M = int(cfg["expand_e"]) * int(cfg["n"]) ** 2
    bad = (i < 0) | (i >= M)
    i[bad] = 0
    ww[bad] = 0.0
    return oracle.lookup_reduce(cfg, t, i, ww)


def _check(cfg, got, want, what):
    err, _ = parity.output_errors(got.float().cpu().numpy(), want)
    assert np.isfinite(got.float().cpu().numpy()).all(), what
    assert err.max() <= parity.out_tol(cfg), f"{what}: {err.max():.3g}"


@pytest.mark.parametrize("name,B,cores", [("decode_1m", 64, 0), ("tiny_fp32", 16, 0),
                                          ("decode_1m", 64, 2)])
def test_noalloc_matches_oracle_and_lookup_reduce_twice(name, B, cores, gpu_lib):
    cfg = workloads.layer_config(name, cores=cores)
    w = workloads.make_weights(cfg, device="cuda")
    layer = binding.UltraMemLayer(cfg, w, B)
    c = _config_struct(cfg, B)
    for call in range(2):   # two calls in a row, different slots each time
        x = workloads.make_tokens(cfg, B, batch_index=call, device="cuda")
        idx, wt = layer.retrieve(x)
        ref = layer.lookup_reduce(idx, wt)
        out = torch.full_like(ref, float("nan"))
        assert _noalloc(gpu_lib, c, w, idx, wt, out) == binding.OK
        torch.cuda.synchronize()
        _check(cfg, out, _oracle_out(cfg, w, idx, wt), f"call {call} vs oracle")
        _check(cfg, out, ref.float().cpu().numpy().astype(np.float64),
               f"call {call} vs lookup_reduce")
    layer.close()


@pytest.mark.parametrize("dtype", [0, 1])
def test_noalloc_explicit_perm_and_bad_addresses(dtype, gpu_lib):
    """A non-null shuffle table, and two addresses outside the grid (one
    past E N, one negative): the output is the oracle's with those slots'
    weights set to 0, on two calls in a row."""
    cfg = workloads.small_config(dtype=dtype, n=10)
    M = cfg["expand_e"] * cfg["n"] ** 2
    perm = torch.from_numpy(np.random.default_rng(5).permutation(M).astype(np.int32)).cuda()
    w = workloads.make_weights(cfg, device="cuda")
    B = 12
    c = _config_struct(cfg, B)
    gen = torch.Generator(device="cpu").manual_seed(9)
    for call in range(2):
        idx = torch.randint(0, M, (B, cfg["heads"], cfg["topm"]), generator=gen,
                            dtype=torch.int64)
        wt = torch.randn((B, cfg["heads"], cfg["topm"]), generator=gen, dtype=torch.float32)
        idx[1, 0, 2] = M + 5
        idx[3 + call, 1, 0] = -1
        idx, wt = idx.cuda(), wt.cuda()
        out = torch.full((B, cfg["d_out"]), float("nan"), dtype=workloads.torch_dtype(cfg),
                         device="cuda")
        assert _noalloc(gpu_lib, c, w, idx, wt, out, perm=perm) == binding.OK
        torch.cuda.synchronize()
        _check(cfg, out, _oracle_out(cfg, w, idx, wt, perm=perm), f"call {call}")


def test_noalloc_after_a_smaller_layer(gpu_lib):
    """A layer created after a no-allocation call must not lower the shared
    memory its kernels were configured for: fp32 rows of 256 at E = 4, then
    a tiny fp32 layer, then the same no-allocation call again."""
    cfg = workloads.small_config(dtype=0, d_v=256, d_out=64, n=12)
    w = workloads.make_weights(cfg, device="cuda")
    B = 8
    c = _config_struct(cfg, B)
    M = cfg["expand_e"] * cfg["n"] ** 2
    gen = torch.Generator(device="cpu").manual_seed(3)
    idx = torch.randint(0, M, (B, cfg["heads"], cfg["topm"]), generator=gen).cuda()
    wt = torch.randn((B, cfg["heads"], cfg["topm"]), generator=gen).cuda()
    want = _oracle_out(cfg, w, idx, wt)
    for step in range(2):
        out = torch.full((B, cfg["d_out"]), float("nan"), device="cuda")
        assert _noalloc(gpu_lib, c, w, idx, wt, out) == binding.OK
        torch.cuda.synchronize()
        _check(cfg, out, want, f"step {step}")
        if step == 0:
            small = workloads.layer_config("tiny_fp32")
            layer = binding.UltraMemLayer(small, workloads.make_weights(small, device="cuda"), 4)
            layer.close()


def test_noalloc_rejects_batches_beyond_its_scratch(gpu_lib):
    cfg = workloads.layer_config("decode_1m")
    c = _config_struct(cfg, 1)
    B = 4096   # needs far more than the static scratch holds
    dummy = torch.zeros(16, dtype=torch.int64, device="cuda")
    st = gpu_lib.ultramem_lookup_reduce_noalloc(C.byref(c), dummy.data_ptr(), dummy.data_ptr(),
                                                None, dummy.data_ptr(), dummy.data_ptr(), B,
                                                dummy.data_ptr(), None)
    assert st == binding.EINVAL
