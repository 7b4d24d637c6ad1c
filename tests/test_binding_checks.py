"""The Python binding's argument checks, on the host (no table is opened: the
checks run before any library call)."""
import pytest
import torch

from paper_2504_01506_gb300.store import EmbeddingStore

CPU = torch.device("cpu")


def _bare(dim=4):
    s = EmbeddingStore.__new__(EmbeddingStore)  # no mlkv_open: the checks need no table
    s.dim = dim
    s.device = CPU
    return s


def test_keys_must_be_1d_int64_on_the_store_device():
    s = _bare()
    k = torch.arange(5, dtype=torch.int64)
    assert s._keys(k).data_ptr() == k.data_ptr()
    for bad in (k.to(torch.int32), k.view(5, 1), k.to(torch.float64)):
        with pytest.raises(TypeError):
            s._keys(bad)
    strided = torch.arange(10, dtype=torch.int64)[::2]
    assert s._keys(strided).is_contiguous() and torch.equal(s._keys(strided), strided)


def test_row_buffers_need_dtype_shape_and_device():
    s = _bare()
    x = torch.zeros(3, 4)
    assert s._rows(x, 3) is x
    for bad, n in ((torch.zeros(3, 5), 3), (torch.zeros(2, 4), 3), (torch.zeros(3, 4, dtype=torch.float64), 3)):
        with pytest.raises(TypeError):
            s._rows(bad, n)


def test_output_buffers_must_be_contiguous():
    """An output is written in place: a strided view would be filled through a
    copy the caller never sees, so it is refused."""
    s = _bare()
    out = torch.zeros(3, 4)
    assert s._check_out(out, 3).data_ptr() == out.data_ptr()
    with pytest.raises(TypeError):
        s._check_out(torch.zeros(4, 3).t(), 3)


def test_host_buffer_calls_check_their_host_tensors():
    s = _bare()
    s.h = None
    with pytest.raises(TypeError):
        s.get_host(torch.arange(3, dtype=torch.int32), torch.zeros(3, 4))      # int32 keys
    with pytest.raises(TypeError):
        s.get_host(torch.arange(3, dtype=torch.int64), torch.zeros(3, 5))      # wrong row width
    with pytest.raises(TypeError):
        s.get_host(torch.arange(3, dtype=torch.int64), torch.zeros(4, 3).t())  # strided output
    with pytest.raises(TypeError):
        s.apply_grad_host(torch.arange(3, dtype=torch.int64), torch.zeros(2, 4))  # one gradient row short
