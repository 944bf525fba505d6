"""Failure paths of the library, made on the host or behind a bounded wait
(no device fault): a bounded mbarrier wait that runs out is reported as
ULTRAMEM_ETIMEOUT and leaves the layer usable; a device allocation that fails
inside ultramem_create is reported as ULTRAMEM_ENOMEM and releases every
allocation the create had made."""
import pytest
import torch

from paper_2411_12364_gb300 import binding, workloads

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("n,B", [(24, 16), (600, 1024)])
def test_bounded_wait_timeout_is_reported_and_next_call_succeeds(n, B, gpu_lib):
    """The scoring kernel's probe (16 tokens: one CTA per tile; 1024 tokens
    on 1200 keys an axis: 160 tiles, the persistent kernel) waits on a
    barrier that nothing signals, gives up after a few thousand cycles and
    records the timeout; the next forward is the normal one again."""
    cfg = workloads.small_config(dtype=1, n=n)
    w = workloads.make_weights(cfg, device="cuda")
    layer = binding.UltraMemLayer(cfg, w, B)
    x = workloads.make_tokens(cfg, B, device="cuda")
    ref = layer.forward(x).clone()
    assert layer.check() == binding.OK
    assert gpu_lib.ultramem_debug_wait_probe(layer._h) == binding.OK
    layer.forward(x)
    assert layer.check() == binding.ETIMEOUT
    assert layer.check() == binding.OK           # the error word was cleared
    out = layer.forward(x)
    assert layer.check() == binding.OK
    assert torch.equal(out, ref)
    layer.close()


def test_wait_probe_needs_the_tensor_core_path(gpu_lib):
    cfg = workloads.small_config(dtype=0)
    layer = binding.UltraMemLayer(cfg, workloads.make_weights(cfg, device="cuda"), 4)
    assert gpu_lib.ultramem_debug_wait_probe(layer._h) == binding.EINVAL
    assert gpu_lib.ultramem_debug_wait_probe(None) == binding.EINVAL
    layer.close()


@pytest.mark.parametrize("dtype", [0, 1])
def test_allocation_failure_returns_enomem_without_leaks(dtype, gpu_lib):
    """Every allocation of ultramem_create in turn fails: the create returns
    ULTRAMEM_ENOMEM and holds nothing afterwards; once the failure lies past
    the create's last allocation, the create succeeds and destroy releases
    everything."""
    cfg = workloads.small_config(dtype=dtype)
    w = workloads.make_weights(cfg, device="cuda")
    base = gpu_lib.ultramem_debug_live_allocations()
    failed = 0
    try:
        for nth in range(64):
            gpu_lib.ultramem_debug_fail_alloc(nth)
            try:
                layer = binding.UltraMemLayer(cfg, w, 40)
            except binding.UltraMemError as e:
                assert e.status == binding.ENOMEM, str(e)
                assert gpu_lib.ultramem_debug_live_allocations() == base
                failed += 1
                continue
            gpu_lib.ultramem_debug_fail_alloc(-1)
            assert gpu_lib.ultramem_debug_live_allocations() > base
            x = workloads.make_tokens(cfg, 40, device="cuda")
            layer.forward(x)
            assert layer.check() == binding.OK
            layer.close()
            assert gpu_lib.ultramem_debug_live_allocations() == base
            break
        else:
            pytest.fail("the create never got past its allocations")
    finally:
        gpu_lib.ultramem_debug_fail_alloc(-1)
    assert failed >= 10   # one failure per workspace buffer
