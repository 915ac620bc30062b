"""The host staging buffer with real registration and copies: fill it from device memory, force
the replacement of one unit (moved aside, fresh pages mapped in place, the buffer registered
again), refill that unit, and read everything back bit for bit."""

import pytest
import torch

from paper_2608_16798_gb300.host_staging import HostStagingBuffer

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def cudart():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    return torch.cuda.cudart()


def test_fill_replace_refill_roundtrip(cudart):
    reg = lambda a, n: cudart.cudaHostRegister(a, n, 0) == cudart.cudaError.success  # noqa: E731
    unreg = lambda a: cudart.cudaHostUnregister(a)  # noqa: E731
    probe_unit = 64 << 20
    buf = HostStagingBuffer(1, reg, unreg, min_unit=probe_unit)  # learn the unit size
    unit = buf.unit
    buf.close()
    nbytes = 2 * unit + unit // 2 + 12_345  # a ragged last unit
    g = torch.Generator(device="cuda").manual_seed(7)
    src = torch.randint(0, 256, (nbytes,), dtype=torch.uint8, device="cuda", generator=g)
    buf = HostStagingBuffer(nbytes, reg, unreg, min_unit=probe_unit)
    try:
        host = torch.frombuffer(buf.buffer(), dtype=torch.uint8)
        host.copy_(src)  # device -> registered host memory
        scratch = torch.empty(buf.unit, dtype=torch.uint8, device="cuda")
        whole = torch.frombuffer(buf.buffer(whole_units=True), dtype=torch.uint8)
        slow_once = {1}

        def probe(off, n):
            scratch[:n].copy_(whole[off:off + n])  # a real copy from the unit
            torch.cuda.synchronize()
            u = off // buf.unit
            if u in slow_once:
                slow_once.discard(u)
                return 1.0
            return 200.0

        def refill(off, n):
            n = max(0, min(n, nbytes - off))
            whole[off:off + n].copy_(src[off:off + n])

        s = buf.qualify(probe, refill)
        assert s["replaced"] == 1 and s["rounds"] == 1 and len(buf.quarantine) == 1
        assert buf.registered
        back = torch.empty_like(src)
        back.copy_(host)  # registered host memory -> device, across the replaced unit
        torch.cuda.synchronize()
        assert torch.equal(back, src)
    finally:
        buf.close()
