"""The read-only stream the kernels' floors are measured with
(stride_selftest_stream_read) reads exactly the bytes it is given: the XOR
of the words it returns, folded over its CTAs, equals the XOR of every 32-bit
word of the buffers computed on the host, for one and two buffers, uneven
slices, and a buffer shorter than the CTAs' threads; bad arguments are
rejected before any launch."""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu


def _xor_words(a: np.ndarray) -> int:
    return int(np.bitwise_xor.reduce(a.view(np.uint32))) if a.size else 0


@pytest.mark.parametrize("nbytes,grid,threads,two", [
    (1 << 20, 152, 128, False),
    (1 << 20, 152, 128, True),
    (16 * 1_000_003, 1024, 128, True),   # slices of uneven length
    (48, 64, 256, True),                 # fewer vectors than threads and CTAs
    (16 * 7919, 3, 1024, False),
])
def test_stream_read_folds_every_word(nbytes, grid, threads, two):
    import torch

    import paper_2609_14636_gb300 as stride

    rng = np.random.default_rng(nbytes % 9973 + grid)
    ha = rng.integers(0, 2**32, nbytes // 4, dtype=np.uint64).astype(np.uint32)
    hb = rng.integers(0, 2**32, nbytes // 4, dtype=np.uint64).astype(np.uint32)
    a = torch.from_numpy(ha.view(np.int32)).cuda()
    b = torch.from_numpy(hb.view(np.int32)).cuda() if two else None
    sink = torch.zeros(grid, dtype=torch.int32, device="cuda")
    stride.stride_selftest_stream_read(a, b, nbytes, grid, threads, sink)
    torch.cuda.synchronize()
    got = _xor_words(sink.cpu().numpy())
    want = _xor_words(ha) ^ (_xor_words(hb) if two else 0)
    assert got == want


def test_stream_read_rejects_bad_arguments():
    import torch

    import paper_2609_14636_gb300 as stride

    a = torch.zeros(1024, dtype=torch.int32, device="cuda")
    sink = torch.zeros(8, dtype=torch.int32, device="cuda")
    L = stride.lib()
    assert L.stride_selftest_stream_read(a.data_ptr(), None, 100, 8, 128, sink.data_ptr(), None) == stride.ERR_INVALID_ARG
    assert L.stride_selftest_stream_read(a.data_ptr() + 4, None, 64, 8, 128, sink.data_ptr(), None) == stride.ERR_INVALID_ARG
    assert L.stride_selftest_stream_read(a.data_ptr(), None, 64, 8, 100, sink.data_ptr(), None) == stride.ERR_INVALID_ARG
    assert L.stride_selftest_stream_read(a.data_ptr(), None, 64, 0, 128, sink.data_ptr(), None) == stride.ERR_INVALID_ARG
    assert L.stride_selftest_stream_read(None, None, 64, 8, 128, sink.data_ptr(), None) == stride.ERR_INVALID_ARG
