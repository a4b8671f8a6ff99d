"""Host-side argument checks of the scoring calls that run before any CUDA
call (CPU only): the vocabulary limit STRIDE_MAX_VOCAB for the batch, step
and shard calls.  An empty window or zero rows returns STRIDE_OK after the
checks, so V = STRIDE_MAX_VOCAB passes them and one column more does not;
the pointers are never dereferenced on these paths."""
import ctypes

import pytest


@pytest.fixture(scope="module")
def lib():
    import paper_2609_14636_gb300 as stride

    return stride, stride.lib()


DUMMY = ctypes.c_void_p(256)  # non-null, aligned; never read: the calls return first


def _batch(L, V, ld):
    d = DUMMY
    return L.stride_score_batch(d, d, 0, ld, V, d, d, d, d, 1, 1, 0, 0, 0, None, -1.0,
                                d, None, None, None, None, d, 1 << 20, None)


def _step(L, V, ld):
    d = DUMMY
    return L.stride_score_step(d, d, 0, ld, V, d, d, 0, 0, None, -1.0, d, None, None, None, None, None)


def _shard(L, V, ld):
    d = DUMMY
    return L.stride_partial_lse(d, d, 0, ld, V, 0, d, 0, d, None, None)


@pytest.mark.parametrize("call", [_batch, _step, _shard])
def test_vocabulary_limit(lib, call):
    stride, L = lib
    V = stride.MAX_VOCAB
    assert call(L, V, V + 8) == stride.OK
    assert call(L, V + 1, V + 8) == stride.ERR_INVALID_ARG
    assert call(L, 0, 8) == stride.ERR_INVALID_ARG
    assert call(L, 16, 15) == stride.ERR_INVALID_ARG  # row stride shorter than a row
