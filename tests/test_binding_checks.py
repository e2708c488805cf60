"""The Python binding's marshalling checks: a call whose tensors are not CUDA
tensors of the format's element type with enough storage is refused before
anything reaches the library, so a caller's mistake cannot send a kernel
outside its buffers.  Runs without a GPU: only refusals are exercised (they
raise before the library is called), with host tensors and with stand-ins
that report themselves as CUDA tensors."""
import pytest
import torch

import paper_2607_12969_gb300 as lrc


class AsCuda:
    """A host tensor presented as a CUDA tensor (on cuda:`index`) to the
    binding's checks."""

    def __init__(self, t, index: int = 0):
        self.t = t
        self.is_cuda = True
        self.device = torch.device("cuda", index)
        self.dtype = t.dtype

    def untyped_storage(self):
        return self.t.untyped_storage()

    def element_size(self):
        return self.t.element_size()

    def storage_offset(self):
        return self.t.storage_offset()

    def numel(self):
        return self.t.numel()

    def half(self):
        return AsCuda(self.t.half(), self.device.index)

    def __getitem__(self, key):
        return AsCuda(self.t[key], self.device.index)


@pytest.fixture(autouse=True)
def current_device_0(monkeypatch):
    """The calls run on cuda:0 (the machine may have no GPU to ask)."""
    monkeypatch.setattr(torch.cuda, "current_device", lambda: 0)


def test_host_tensors_are_refused():
    U = torch.zeros((4, 16), dtype=torch.float32)
    with pytest.raises(ValueError, match="CUDA tensor"):
        lrc.lrc_apply(U, U, U, U, U, 4, 4, 2, 1, "f32")
    with pytest.raises(ValueError, match="CUDA tensor"):
        lrc.tt_reconstruct([torch.zeros(6)], [6], [1, 1], "f32", torch.zeros(6))
    with pytest.raises(ValueError, match="CUDA tensor"):
        lrc.lrc_fro_diff(torch.zeros(8, dtype=torch.float64), "f64", None, "f64", 8)
    with pytest.raises(ValueError, match="CUDA tensor"):
        lrc.lrc_round_factors(torch.zeros((2, 3), dtype=torch.float64), 2, 3, 3,
                              torch.zeros((2, 16), dtype=torch.float32), 16, "f32")
    with pytest.raises(ValueError, match="a tensor is required"):
        lrc.lrc_apply(None, U, U, U, U, 4, 4, 2, 1, "f32")


def test_extent_of_a_pitched_array():
    assert lrc._extent(3, 5, 16) == 2 * 16 + 5
    assert lrc._extent(0, 5, 16) == 0 and lrc._extent(3, 0, 16) == 0


def test_wrong_type_or_short_storage_is_refused():
    m, n, k, b = 64, 48, 8, 5
    ldk, ldn = 16, 48
    h = lambda shape, dt: AsCuda(torch.zeros(shape, dtype=dt))       # noqa: E731
    U, S = h((m, ldk), torch.float16), h((1, ldk), torch.float16)
    Vt, X = h((k, ldn), torch.float16), h((b, ldn), torch.float16)
    Y = h((b, m), torch.float32)
    with pytest.raises(ValueError, match="element type"):
        lrc.lrc_apply(U, S, Vt, X, Y.half(), m, n, k, b, "f16")         # F16 writes binary32
    with pytest.raises(ValueError, match="storage holds"):
        lrc.lrc_apply(U, S, Vt, X, Y[:, 1:], m, n, k, b, "f16")         # a view one element short
    with pytest.raises(ValueError, match="storage holds"):
        lrc.lrc_apply(h((m - 1, ldk), torch.float16), S, Vt, X, Y, m, n, k, b, "f16")   # a row of U missing
    with pytest.raises(ValueError, match="element type"):
        lrc.lrc_apply(U, S, Vt, h((b, ldn), torch.float32), Y, m, n, k, b, "f16")     # X in binary32
    cores = [h((1, 6, 2), torch.float32), h((2, 5, 1), torch.float32)]
    with pytest.raises(ValueError, match="storage holds"):
        lrc.tt_reconstruct(cores, [6, 5], [1, 2, 1], "f32", h((29,), torch.float32))
    with pytest.raises(ValueError, match="storage holds"):
        lrc.tt_reconstruct([h((1, 6, 2), torch.float32), h((2, 4, 1), torch.float32)], [6, 5], [1, 2, 1], "f32",
                           h((30,), torch.float32))
    with pytest.raises(ValueError, match="storage holds"):
        lrc.lrc_fro_diff(h((99,), torch.float64), "f64", None, "f64", 100)


def test_views_are_measured_from_their_first_element():
    base = torch.zeros((5, 64))
    assert lrc._span(base[:, 1:]) == 5 * 64 - 1
    assert lrc._span(base[1:]) == 4 * 64


def test_tensor_on_another_gpu_is_refused():
    """A tensor on cuda:1 passed to a call that runs on cuda:0 would hand a
    kernel a pointer into another GPU's memory: it is refused."""
    m, n, k, b = 64, 48, 8, 5
    h = lambda shape, dt, i=0: AsCuda(torch.zeros(shape, dtype=dt), i)    # noqa: E731
    U, S = h((m, 16), torch.float32), h((1, 16), torch.float32)
    Vt, X, Y = h((k, n), torch.float32), h((b, n), torch.float32), h((b, m), torch.float32)
    with pytest.raises(ValueError, match="cuda:1"):
        lrc.lrc_apply(U, S, Vt, h((b, n), torch.float32, 1), Y, m, n, k, b, "f32")
    with pytest.raises(ValueError, match="cuda:1"):
        lrc.lrc_apply(U, S, Vt, X, h((b, m), torch.float32, 1), m, n, k, b, "f32")
    with pytest.raises(ValueError, match="cuda:1"):
        lrc.tt_reconstruct([h((1, 6, 2), torch.float32), h((2, 5, 1), torch.float32, 1)], [6, 5], [1, 2, 1],
                           "f32", h((30,), torch.float32))
    with pytest.raises(ValueError, match="cuda:1"):
        lrc.lrc_fro_diff(h((100,), torch.float64), "f64", h((100,), torch.float64, 1), "f64", 100)

    class OnDevice1:
        device = torch.device("cuda", 1)
        cuda_stream = 0
    # a stream of cuda:1 with tensors on cuda:0
    with pytest.raises(ValueError, match="cuda:0, but the call runs on cuda:1"):
        lrc.lrc_fro_diff(h((100,), torch.float64), "f64", None, "f64", 100, stream=OnDevice1())
