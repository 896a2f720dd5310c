import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built library")


def pytest_collection_modifyitems(config, items):
    try:
        import torch

        has_gpu = torch.cuda.is_available()
    except Exception:  # pragma: no cover
        has_gpu = False
    if has_gpu:
        return
    skip = pytest.mark.skip(reason="no CUDA device")
    for item in items:
        if "gpu" in item.keywords:
            item.add_marker(skip)


# ------------------------------------------------------------------ guard canaries
#
# Every device buffer a GPU test allocates with torch.empty / torch.zeros /
# torch.full (outputs, result blocks and workspaces, which the binding's
# make_result / make_workspace allocate the same way) sits between two 4 KB
# canary regions of a known byte pattern; after the test the canaries must be
# intact, so a kernel that writes before or past the end of any buffer fails
# the test that ran it.  Buffers above 64 MB (the full-size caches and weights,
# whose every byte the tests compare anyway) are allocated plainly.

GUARD_BYTES = 4096
GUARD_MAX_BYTES = 64 << 20
CANARY = 0xA5


class _Guards:
    def __init__(self, torch):
        self.torch = torch
        self.orig = {name: getattr(torch, name) for name in ("empty", "zeros", "full")}
        self.bufs = []

    @staticmethod
    def _shape(args, size_kw):
        if size_kw is not None:
            args = (size_kw,)
        if len(args) == 1 and not isinstance(args[0], int):
            return tuple(int(x) for x in args[0])
        return tuple(int(x) for x in args)

    def _guarded(self, shape, dtype, device):
        torch = self.torch
        n = 1
        for x in shape:
            n *= x
        nbytes = n * dtype.itemsize
        buf = self.orig["empty"](nbytes + 2 * GUARD_BYTES, dtype=torch.uint8, device=device)
        buf[:GUARD_BYTES].fill_(CANARY)
        buf[GUARD_BYTES + nbytes:].fill_(CANARY)
        self.bufs.append((buf, nbytes))
        return buf[GUARD_BYTES:GUARD_BYTES + nbytes].view(dtype).view(shape)

    def _eligible(self, shape, kw):
        torch = self.torch
        dev = kw.get("device")
        if dev is None or torch.device(dev).type != "cuda":
            return False
        if set(kw) - {"dtype", "device"}:
            return False
        n = 1
        for x in shape:
            n *= x
        return n * (kw.get("dtype") or torch.get_default_dtype()).itemsize <= GUARD_MAX_BYTES

    def install(self):
        torch = self.torch

        def empty(*args, size=None, **kw):
            shape = self._shape(args, size)
            if not self._eligible(shape, kw):
                return self.orig["empty"](*args, **({"size": size} if size is not None else {}), **kw)
            return self._guarded(shape, kw.get("dtype") or torch.get_default_dtype(), kw["device"])

        def zeros(*args, size=None, **kw):
            shape = self._shape(args, size)
            if not self._eligible(shape, kw):
                return self.orig["zeros"](*args, **({"size": size} if size is not None else {}), **kw)
            return self._guarded(shape, kw.get("dtype") or torch.get_default_dtype(), kw["device"]).zero_()

        def full(size, fill_value, **kw):
            shape = self._shape((size,), None)
            if not self._eligible(shape, kw):
                return self.orig["full"](size, fill_value, **kw)
            return self._guarded(shape, kw.get("dtype") or torch.get_default_dtype(), kw["device"]).fill_(fill_value)

        torch.empty, torch.zeros, torch.full = empty, zeros, full

    def uninstall(self):
        for name, fn in self.orig.items():
            setattr(self.torch, name, fn)

    def check(self):
        torch = self.torch
        if torch.cuda.is_available():
            torch.cuda.synchronize()
        bad = []
        for buf, nbytes in self.bufs:
            head, tail = buf[:GUARD_BYTES], buf[GUARD_BYTES + nbytes:]
            if bool((head != CANARY).any()) or bool((tail != CANARY).any()):
                bad.append(nbytes)
        self.bufs.clear()
        return bad


@pytest.fixture(autouse=True)
def guard_canaries(request):
    if "gpu" not in request.keywords:
        yield
        return
    import torch

    if not torch.cuda.is_available():
        yield
        return
    guards = _Guards(torch)
    guards.install()
    try:
        yield
    finally:
        guards.uninstall()
    bad = guards.check()
    assert not bad, f"a kernel wrote outside {len(bad)} device buffer(s) of {bad} bytes (guard canaries overwritten)"
    if os.environ.get("TB_DEBUG_BOUNDS") == "1":
        # the debug build of the library: no kernel may have failed an index check
        import paper_2606_27550_gb300 as tv

        n = tv.tb_debug_bounds_violations()
        assert n == 0, f"{n} global-memory index checks failed in the debug build"
