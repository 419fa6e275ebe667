"""GPU test of duo_pack_cmb_noalloc, the packing entry point that allocates
nothing (for callers that cannot call cudaMalloc themselves).

It must produce exactly the bytes of duo_pack, on two calls in a row (the
calls share one static scratch array), and reject what exceeds its limits.
This file is collected last so that a run stopping at the first failure has
run every other test already; it also passes when run alone.
"""
import ctypes

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def duo():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2506_20194_gb300 import duo as d
    d.load_library()
    return d


def _weight(O, I, seed, pw=0.5):
    g = torch.Generator().manual_seed(seed)
    W = (torch.randn(O, I, generator=g) * 0.02).to(torch.float16)
    W[torch.rand(O, I, generator=g) < pw] = 0
    return W.cuda()


def test_noalloc_pack_matches_duo_pack_twice(duo):
    # Two different weights packed one after the other: the second call reuses
    # the scratch the first one filled.
    for W in (_weight(2100, 333, 1), _weight(4096, 1000, 2, pw=0.3)):
        O, I = W.shape
        off, data, nbytes = duo.duo_pack_cmb_noalloc(W)
        h = duo.duo_pack(W, "bitmask")
        info, ref_off, _, ref_data = duo.packed_bytes(h)
        assert nbytes == info.data_bytes
        assert np.array_equal(off.cpu().numpy().view(np.uint8), ref_off)
        assert np.array_equal(data[:nbytes].cpu().numpy(), ref_data)
        h.free()
    assert duo.duo_device_status() == duo.DUO_OK


def test_noalloc_limits_and_size_query(duo):
    lib = duo.load_library()
    W = _weight(1500, 200, 3)
    O, I = W.shape
    S = (O + 1023) // 1024
    off = torch.empty(I * S + 1, dtype=torch.int32, device="cuda")
    nb = ctypes.c_int64(-1)
    stream = torch.cuda.current_stream().cuda_stream
    # size query (no data buffer), then a too-small buffer
    assert lib.duo_pack_cmb_noalloc(W.data_ptr(), O, I, I, off.data_ptr(), None, 0,
                                    ctypes.byref(nb), stream) == duo.DUO_OK
    need = nb.value
    small = torch.empty(16, dtype=torch.uint8, device="cuda")
    nb2 = ctypes.c_int64(-1)
    assert lib.duo_pack_cmb_noalloc(W.data_ptr(), O, I, I, off.data_ptr(), small.data_ptr(), 16,
                                    ctypes.byref(nb2), stream) == duo.DUO_ERANGE
    assert nb2.value == need
    # beyond the scratch limit: in * ceil(out / 1024) > DUO_NOALLOC_MAX_RECORDS
    big_in = 65535
    big_out = 1024 * 5            # 5 segments x 65535 channels > 262144 records
    assert lib.duo_pack_cmb_noalloc(W.data_ptr(), big_out, big_in, big_in, off.data_ptr(),
                                    small.data_ptr(), 16, ctypes.byref(nb2), stream) == duo.DUO_ERANGE


def test_noalloc_rejects_before_device_work(duo):
    lib = duo.load_library()
    W = _weight(64, 8, 4)
    off = torch.empty(64, dtype=torch.int32, device="cuda")
    data = torch.empty(4096, dtype=torch.uint8, device="cuda")
    nb = ctypes.c_int64(-1)
    stream = torch.cuda.current_stream().cuda_stream
    # more than 65535 segments: in = 1 keeps the record count under the limit
    assert lib.duo_pack_cmb_noalloc(W.data_ptr(), 65536 * 1024, 1, 1, off.data_ptr(),
                                    data.data_ptr(), 4096, ctypes.byref(nb), stream) == duo.DUO_ERANGE
    # host memory where device memory is required
    host_off = np.zeros(64, dtype=np.uint32)
    host_data = np.zeros(4096 + 16, dtype=np.uint8)
    hd = host_data.ctypes.data + (-host_data.ctypes.data) % 16
    assert lib.duo_pack_cmb_noalloc(W.data_ptr(), 64, 8, 8, host_off.ctypes.data,
                                    data.data_ptr(), 4096, ctypes.byref(nb), stream) == duo.DUO_EINVAL
    assert lib.duo_pack_cmb_noalloc(W.data_ptr(), 64, 8, 8, off.data_ptr(),
                                    hd, 4096, ctypes.byref(nb), stream) == duo.DUO_EINVAL
    assert duo.duo_device_status() == duo.DUO_OK


def test_noalloc_allocates_no_device_memory(duo):
    """The point of the entry point: with every buffer allocated beforehand,
    a call leaves the device's free memory unchanged."""
    lib = duo.load_library()
    W = _weight(3000, 700, 5)
    O, I = W.shape
    S = (O + 1023) // 1024
    off = torch.empty(I * S + 1, dtype=torch.int32, device="cuda")
    nb = ctypes.c_int64(-1)
    stream = torch.cuda.current_stream().cuda_stream
    assert lib.duo_pack_cmb_noalloc(W.data_ptr(), O, I, I, off.data_ptr(), None, 0,
                                    ctypes.byref(nb), stream) == duo.DUO_OK
    data = torch.empty(nb.value, dtype=torch.uint8, device="cuda")
    call = lambda: lib.duo_pack_cmb_noalloc(W.data_ptr(), O, I, I, off.data_ptr(), data.data_ptr(),
                                            nb.value, ctypes.byref(nb), stream)
    assert call() == duo.DUO_OK   # warm-up: module load and first-call set-up
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    for _ in range(3):
        assert call() == duo.DUO_OK
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0
