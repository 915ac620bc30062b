"""Page-locked host memory for streaming a step's inputs to the GPU.

One anonymous mapping, aligned to and advised for transparent huge pages, touched, then
registered with the CUDA runtime. Its units (a whole number of huge pages, at least
``min_unit`` bytes) can be qualified: a caller-supplied probe times a host-to-device copy
from each unit, and units well below the median are moved out of the way (``mremap``; they
stay allocated until ``close()`` so that the kernel cannot hand the same physical pages back)
and replaced in place by fresh pages, which the caller refills. The virtual addresses never
change, so the whole buffer stays one registered range that a single copy can read from end to
end.

On virtual machines, a few physical huge pages can be much slower sources of device reads
than the rest (3-72 GB/s against 210 GB/s from the others, measured on GB300 hosts): which
pages are slow changes from one process to the next, stays the same within it once the data is
written, and can change when the buffer is first written. Qualification costs one copy per unit
and runs after the buffer is filled, before any timed work.

The memory calls are made through libc with ctypes (Linux only); registration and the probe
are injected, so the logic runs without a GPU.
"""

from __future__ import annotations

import ctypes
import mmap
import os
import statistics

import numpy as np

_PROT_RW = mmap.PROT_READ | mmap.PROT_WRITE
_MAP_FIXED = 0x10  # same value on x86-64 and aarch64 Linux
_MREMAP_MAYMOVE = 1
_MREMAP_FIXED = 2
_MAP_FAILED = ctypes.c_void_p(-1).value

_libc = None


def _lib():
    global _libc
    if _libc is None:
        lib = ctypes.CDLL(None, use_errno=True)
        lib.mmap.restype = ctypes.c_void_p
        lib.mmap.argtypes = [ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                             ctypes.c_long]
        lib.munmap.restype = ctypes.c_int
        lib.munmap.argtypes = [ctypes.c_void_p, ctypes.c_size_t]
        lib.madvise.restype = ctypes.c_int
        lib.madvise.argtypes = [ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int]
        lib.mremap.restype = ctypes.c_void_p
        # the fifth (variadic) argument, the new address, is read only with MREMAP_FIXED
        lib.mremap.argtypes = [ctypes.c_void_p, ctypes.c_size_t, ctypes.c_size_t, ctypes.c_int, ctypes.c_void_p]
        _libc = lib
    return _libc


def huge_page_size() -> int:
    """The transparent huge page size (2 MiB on x86-64, 512 MiB on aarch64 with 64 KiB pages)."""
    try:
        with open("/sys/kernel/mm/transparent_hugepage/hpage_pmd_size") as f:
            return int(f.read().strip())
    except (OSError, ValueError):
        return 2 << 20


def _check_map(addr, what):
    if addr is None or addr == _MAP_FAILED:
        err = ctypes.get_errno()
        raise OSError(err, f"{what}: {os.strerror(err)}")
    return addr


class HostStagingBuffer:
    """``nbytes`` of page-locked host memory at a fixed address, optionally qualified.

    register(addr, nbytes) -> bool and unregister(addr) pin and unpin the range (for CUDA:
    cudaHostRegister / cudaHostUnregister); None leaves the memory pageable.
    """

    def __init__(self, nbytes: int, register=None, unregister=None, min_unit: int = 256 << 20):
        if nbytes <= 0:
            raise ValueError("nbytes must be positive")
        lib = _lib()
        self.hp = huge_page_size()
        self.page = mmap.PAGESIZE
        self.unit = max(self.hp, -(-min_unit // self.hp) * self.hp)
        self.nbytes = nbytes
        self.size = -(-nbytes // self.unit) * self.unit  # whole units
        self._register, self._unregister = register, unregister
        self.quarantine: list[tuple[int, int]] = []
        self.replaced = 0
        self.rounds = 0
        self.unit_gbs: list[float] = []
        self.registered = False
        self.broken = False  # set if a failed replacement left part of the range unmapped
        # reserve size + one huge page, keep the aligned part
        raw = _check_map(lib.mmap(None, self.size + self.hp, _PROT_RW, mmap.MAP_PRIVATE | mmap.MAP_ANONYMOUS, -1, 0),
                         "mmap")
        base = -(-raw // self.hp) * self.hp
        if base > raw:
            lib.munmap(raw, base - raw)
        tail = raw + self.size + self.hp - (base + self.size)
        if tail > 0:
            lib.munmap(base + self.size, tail)
        self.addr = base
        self._prepare(0, self.size)
        self._pin()

    # -- memory ---------------------------------------------------------------------------------
    def _prepare(self, off, length):
        """Advise huge pages for [off, off + length) and touch every base page of it."""
        lib = _lib()
        if hasattr(mmap, "MADV_HUGEPAGE"):
            lib.madvise(self.addr + off, length, mmap.MADV_HUGEPAGE)
        view = np.frombuffer((ctypes.c_uint8 * length).from_address(self.addr + off), dtype=np.uint8)
        view[::self.page] = 0

    def _pin(self):
        if self._register is not None and not self.registered:
            if not self._register(self.addr, self.size):
                raise RuntimeError("registering the host staging buffer was refused")
            self.registered = True

    def _unpin(self):
        if self.registered:
            self._unregister(self.addr)
            self.registered = False

    def _replace(self, units):
        """Move the given units out of the way (kept allocated) and map fresh pages in place.
        The buffer is registered again even when a step fails (the error is then raised)."""
        lib = _lib()
        self._unpin()
        try:
            for u in units:
                off = u * self.unit
                # a same-size mremap without a destination is a no-op: reserve one and move there
                dest = _check_map(lib.mmap(None, self.unit, 0, mmap.MAP_PRIVATE | mmap.MAP_ANONYMOUS, -1, 0),
                                  "mmap")
                moved = lib.mremap(self.addr + off, self.unit, self.unit, _MREMAP_MAYMOVE | _MREMAP_FIXED, dest)
                if moved is None or moved == _MAP_FAILED:
                    err = ctypes.get_errno()
                    lib.munmap(dest, self.unit)
                    raise OSError(err, f"mremap: {os.strerror(err)}")
                # the unit's range is unmapped now: map fresh pages there, or put the old ones back
                got = lib.mmap(self.addr + off, self.unit, _PROT_RW,
                               mmap.MAP_PRIVATE | mmap.MAP_ANONYMOUS | _MAP_FIXED, -1, 0)
                if got != self.addr + off:
                    err = ctypes.get_errno()
                    back = lib.mremap(moved, self.unit, self.unit, _MREMAP_MAYMOVE | _MREMAP_FIXED, self.addr + off)
                    if back != self.addr + off:
                        self.broken = True  # a hole in the buffer: it must not be used any more
                        self.quarantine.append((moved, self.unit))
                    raise OSError(err, f"mmap fixed: {os.strerror(err)}")
                self.quarantine.append((moved, self.unit))
                self._prepare(off, self.unit)
                self.replaced += 1
        finally:
            if not self.broken:
                self._pin()

    # -- qualification --------------------------------------------------------------------------
    @property
    def n_units(self) -> int:
        return self.size // self.unit

    def qualify(self, probe, refill=None, slow_frac: float = 0.6, max_rounds: int = 4) -> dict:
        """Time each unit with probe(offset, nbytes) -> GB/s; replace units below slow_frac x the
        median, call refill(offset, nbytes) for each replaced unit (its fresh pages read as zero),
        and probe them again, at most max_rounds times. Returns a summary.

        Qualify a buffer after writing its contents: on the hosts measured, pages that copied fast
        while untouched could turn slow once the buffer was first written."""
        gbs = [float(probe(u * self.unit, self.unit)) for u in range(self.n_units)]
        ref = statistics.median(gbs)
        for _ in range(max_rounds):
            slow = [u for u in range(self.n_units) if gbs[u] < slow_frac * ref]
            if not slow:
                break
            self.rounds += 1
            self._replace(slow)
            for u in slow:
                if refill is not None:
                    refill(u * self.unit, self.unit)
                gbs[u] = float(probe(u * self.unit, self.unit))
        self.unit_gbs = gbs
        return self.summary()

    def summary(self) -> dict:
        g = self.unit_gbs
        return {"unit_bytes": self.unit, "units": self.n_units, "replaced": self.replaced, "rounds": self.rounds,
                "unit_gbs_min": min(g) if g else None, "unit_gbs_median": statistics.median(g) if g else None}

    # -- access ---------------------------------------------------------------------------------
    def buffer(self, whole_units: bool = False):
        """A ctypes array (it supports the buffer protocol) over the first nbytes, or over every
        unit with whole_units. It is valid until close()."""
        if self.addr is None or self.broken:
            raise ValueError("the buffer is closed" if self.addr is None else "the buffer has a hole")
        return (ctypes.c_uint8 * (self.size if whole_units else self.nbytes)).from_address(self.addr)

    def close(self):
        if self.addr is None:
            return
        lib = _lib()
        self._unpin()
        lib.munmap(self.addr, self.size)  # unmapping a range with a hole in it is fine
        for a, n in self.quarantine:
            lib.munmap(a, n)
        self.quarantine = []
        self.addr = None

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()
