"""ultramem_lookup_reduce_noalloc: the lookup-reduce for callers that cannot
allocate device memory (no layer handle, scratch in static device memory).
Its output must match the handle-based ultramem_lookup_reduce on the same
slots, on two calls in a row (the static scratch keeps the previous call's
contents).  Collected last so that a failure here cannot hide the others."""
import ctypes as C

import numpy as np
import pytest
import torch

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


def _noalloc(lib, c, w, idx, wt, out):
    st = lib.ultramem_lookup_reduce_noalloc(
        C.byref(c), w["values"].data_ptr(),
        None if w.get("w_proj") is None else w["w_proj"].data_ptr(), None,
        idx.data_ptr(), wt.data_ptr(), idx.shape[0], out.data_ptr(),
        torch.cuda.current_stream().cuda_stream)
    return st


@pytest.mark.parametrize("name,B,cores", [("decode_1m", 64, 0), ("tiny_fp32", 16, 0),
                                          ("decode_1m", 64, 2)])
def test_noalloc_matches_lookup_reduce_twice(name, B, cores, gpu_lib):
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
        got = out.float().cpu().numpy().astype(np.float64)
        want = ref.float().cpu().numpy().astype(np.float64)
        err = np.abs(got - want).max(1) / np.maximum(np.abs(want).max(1), 1e-30)
        assert np.isfinite(got).all()
        assert err.max() <= parity.out_tol(cfg), f"call {call}: {err.max()}"
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
