"""The guard canaries of the GPU tests (tests/conftest.py), exercised on host
tensors: a write one byte before or past a guarded buffer is reported, writes
inside it are not, and the allocation wrappers give the requested shapes,
dtypes and fill values."""
import torch

import conftest


def _guards():
    return conftest._Guards(torch)


def test_untouched_and_inside_writes_pass():
    g = _guards()
    t = g._guarded((3, 5), torch.float32, "cpu")
    t.fill_(7.0)
    t[-1, -1] = -1.0
    assert t.shape == (3, 5) and t.dtype == torch.float32 and t.is_contiguous()
    assert g.check() == []


def test_write_past_the_end_is_reported():
    g = _guards()
    t = g._guarded((16,), torch.int32, "cpu")
    buf, nbytes = g.bufs[-1]
    buf[conftest.GUARD_BYTES + nbytes] = 0  # the first byte after the buffer
    assert g.check() == [16 * 4]


def test_write_before_the_start_is_reported():
    g = _guards()
    g._guarded((2, 2), torch.bfloat16, "cpu")
    buf, _ = g.bufs[-1]
    buf[conftest.GUARD_BYTES - 1] = 0  # the last byte before the buffer
    assert len(g.check()) == 1


def test_wrapper_shapes_and_fill():
    g = _guards()
    assert g._shape((4,), None) == (4,)
    assert g._shape(((2, 3),), None) == (2, 3)
    assert g._shape((2, 3), None) == (2, 3)
    assert g._shape((), torch.Size([5])) == (5,)
    # only device allocations without extra options are guarded
    assert not g._eligible((4,), {"dtype": torch.float32})
    assert not g._eligible((4,), {"dtype": torch.float32, "device": "cpu"})
    assert not g._eligible((4,), {"dtype": torch.float32, "device": "cuda", "pin_memory": True})
    assert g._eligible((4,), {"dtype": torch.float32, "device": "cuda"})
    assert not g._eligible((1 << 30,), {"dtype": torch.float32, "device": "cuda"})
