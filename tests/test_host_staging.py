"""The host staging buffer: alignment, qualification and replacement of slow units (CPU only;
a fake probe stands in for the device copy and registration is a recording fake)."""

import ctypes

import numpy as np
import pytest

from paper_2608_16798_gb300.host_staging import HostStagingBuffer, huge_page_size


def _arr(buf, whole=False):
    return np.frombuffer(buf.buffer(whole), dtype=np.uint8)


def test_layout_and_registration():
    events = []
    reg = lambda a, n: events.append(("reg", a, n)) or True
    unreg = lambda a: events.append(("unreg", a))
    b = HostStagingBuffer(3 * (4 << 20) + 5, reg, unreg, min_unit=4 << 20)
    try:
        hp = huge_page_size()
        assert b.addr % hp == 0 and b.unit % hp == 0 and b.unit >= 4 << 20
        assert b.size % b.unit == 0 and b.size >= b.nbytes
        assert events == [("reg", b.addr, b.size)]
        a = _arr(b)
        assert a.size == b.nbytes and not a.any()  # fresh anonymous pages read as zero
        a[:] = 3
        assert int(a.sum()) == 3 * b.nbytes
    finally:
        b.close()
    assert events[-1] == ("unreg", events[0][1])
    with pytest.raises(ValueError):
        b.buffer()


def test_qualification_replaces_only_slow_units():
    events = []
    b = HostStagingBuffer(6 * (4 << 20), lambda a, n: events.append("reg") or True,
                          lambda a: events.append("unreg"), min_unit=4 << 20)
    try:
        n, unit, addr = b.n_units, b.unit, b.addr
        full = _arr(b, whole=True)
        for u in range(n):
            full[u * unit:(u + 1) * unit] = u + 1  # a pattern per unit
        stays_slow = {1: 1, 3: 2}  # unit -> number of probes that still read slow
        calls = []

        def probe(off, nbytes):
            assert nbytes == unit and off % unit == 0
            u = off // unit
            calls.append(("probe", u))
            if stays_slow.get(u, 0):
                stays_slow[u] -= 1
                return 12.0
            return 210.0

        def refill(off, nbytes):
            u = off // unit
            fresh = _arr(b, whole=True)[off:off + nbytes]
            assert not fresh.any(), "a replaced unit starts with fresh (zero) pages"
            fresh[:] = 100 + u
            calls.append(("refill", u))

        s = b.qualify(probe, refill)
        assert calls == [("probe", u) for u in range(n)] + [
            ("refill", 1), ("probe", 1), ("refill", 3), ("probe", 3), ("refill", 3), ("probe", 3)]
        assert s["replaced"] == 3 and s["rounds"] == 2 and s["unit_gbs_min"] == 210.0
        assert b.addr == addr and events == ["reg", "unreg", "reg", "unreg", "reg"]
        full = _arr(b, whole=True)
        for u in range(n):  # replaced units hold the refilled data, the others kept theirs
            want = 100 + u if u in (1, 3) else u + 1
            assert (full[u * unit:(u + 1) * unit] == want).all(), u
        # the pages moved out are still mapped, with their data, outside the buffer
        assert len(b.quarantine) == 3
        # (units 1 and 3 held their patterns in the first round; unit 3 its refill in the second)
        for (qa, qn), want in zip(b.quarantine, (2, 4, 103)):
            assert not (addr <= qa < addr + b.size) and qn == unit
            q = np.frombuffer((ctypes.c_uint8 * qn).from_address(qa), dtype=np.uint8)
            assert (q == want).all()
    finally:
        b.close()
    assert b.quarantine == []


def test_uniform_units_are_left_alone():
    b = HostStagingBuffer(2 * (4 << 20), min_unit=4 << 20)
    try:
        s = b.qualify(lambda off, n: 200.0 + (off // b.unit))
        assert s["replaced"] == 0 and s["rounds"] == 0 and not b.quarantine
    finally:
        b.close()


def test_refused_registration_raises_and_rejects_bad_size():
    with pytest.raises(ValueError):
        HostStagingBuffer(0)
    with pytest.raises(RuntimeError):
        HostStagingBuffer(1 << 20, lambda a, n: False, lambda a: None)


def test_failed_replacement_registers_again(monkeypatch):
    """A replacement whose fresh mapping is refused puts the old pages back, registers the
    buffer again and raises; the data and the addresses are unchanged."""
    import paper_2608_16798_gb300.host_staging as HS

    events = []
    b = HostStagingBuffer(3 * (4 << 20), lambda a, n: events.append("reg") or True,
                          lambda a: events.append("unreg"), min_unit=4 << 20)
    try:
        full = _arr(b, whole=True)
        full[:] = 9
        lib = HS._lib()
        real_mmap = lib.mmap

        class Refusing:  # refuses MAP_FIXED requests, passes the others through
            def __call__(self, addr, length, prot, flags, fd, off):
                if flags & HS._MAP_FIXED:
                    ctypes.set_errno(12)
                    return HS._MAP_FAILED
                return real_mmap(addr, length, prot, flags, fd, off)

        monkeypatch.setattr(lib, "mmap", Refusing())
        with pytest.raises(OSError):
            b.qualify(lambda off, n: 1.0 if off // b.unit == 1 else 200.0)
        monkeypatch.setattr(lib, "mmap", real_mmap)
        assert not b.broken and b.registered and events[-1] == "reg"
        assert (_arr(b, whole=True) == 9).all()  # the old pages are back in place
        assert b.quarantine == []
    finally:
        b.close()
