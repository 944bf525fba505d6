"""The per-stage profiling of the library: each kernel of a forward stamps
the GPU's global timer, also when the forward is captured in a CUDA graph and
replayed (the bench's stage times and roofline come from these)."""
import pytest
import torch

from paper_2411_12364_gb300 import binding, workloads

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("dtype", [0, 1])
def test_stage_stamps_cover_the_forward(dtype, gpu_lib):
    cfg = workloads.small_config(dtype=dtype)
    layer = binding.UltraMemLayer(cfg, workloads.make_weights(cfg, device="cuda"), 40)
    x = workloads.make_tokens(cfg, 40, device="cuda")
    ref = layer.forward(x).clone()
    assert layer.profile_read() == {}            # nothing profiled yet
    layer.profile(True)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        out = layer.forward(x)
        torch.cuda.synchronize()
        t, g = layer.profile_read(gaps=True)
        assert set(t) == {"query", "score", "select", "gather", "project"}
        assert all(v > 0 for v in t.values()), t
        assert all(v >= 0 for v in g.values()) and g["query"] == 0, g
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=s):
            layer.forward(x, out=out)
        for _ in range(2):
            out.zero_()
            graph.replay()
            torch.cuda.synchronize()
            t2 = layer.profile_read()
            assert all(v > 0 for v in t2.values()), t2
            assert torch.equal(out, ref)         # the stamps change no result
    layer.profile(False)
    assert layer.check() == binding.OK
    layer.close()
