"""GPU parity of the quantised-value path (§5, weight-only quantisation with
channel-wise RTN and group size 128, Table 4) through the C ABI against the
CPU oracle.

Bar: packed records, offsets and grid tables bit-exact against the oracle's
packer; y within 2e-3 * sum_{j in K} |W_hat_ij| |x_j| per row (W_hat the
dequantised weight), and exactly 0 where that sum is 0.
"""
import numpy as np
import pytest
import torch

import oracle as orc

pytestmark = pytest.mark.gpu

REL_TOL = 2e-3
FMT = {8: "bitmask_q8", 4: "bitmask_q4"}


@pytest.fixture(scope="module")
def duo():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2506_20194_gb300 import duo as d
    d.load_library()
    return d


def _np16(t):
    return t.detach().cpu().numpy().view(np.float16)


def _laplace(I, seed):
    g = torch.Generator().manual_seed(seed)
    u = torch.rand(I, generator=g, dtype=torch.float64) - 0.5
    return (-torch.sign(u) * torch.log1p(-2 * u.abs())).to(torch.float16)


def _weight(O, I, pw, seed, kind="gauss"):
    g = torch.Generator().manual_seed(seed)
    if kind == "gauss":
        W = (torch.randn(O, I, generator=g) * 0.02).to(torch.float16)
    elif kind == "halves":        # on power-of-two grids: half-way cases for RTN
        W = (torch.randint(-8, 9, (O, I), generator=g) * 0.125).to(torch.float16)
    elif kind == "onesided":      # whole groups of one sign
        W = (torch.randn(O, I, generator=g).abs() * 0.05).to(torch.float16)
        W[: O // 2] = -W[: O // 2]
    else:                         # wide range, subnormals included
        e = torch.randint(-22, 4, (O, I), generator=g).to(torch.float32)
        W = (torch.randn(O, I, generator=g) * torch.pow(2.0, e)).to(torch.float16)
    W[torch.rand(O, I, generator=g) < pw] = 0
    if O > 2:
        W[1] = 0                  # a row with no stored weight: empty groups
    return W


def _check_y(y_gpu, Wd, x16, K, label):
    xv = x16.astype(np.float64)
    Kl = np.asarray(K, dtype=np.int64)
    y_ref = Wd[:, Kl] @ xv[Kl]
    tol = orc.tolerance_rows_f64(Wd, x16, K, REL_TOL)
    y = np.asarray(y_gpu, dtype=np.float64)
    err = np.abs(y - y_ref)
    bad = err > tol
    assert not bad.any(), (f"{label}: {bad.sum()} rows out of tolerance; worst row "
                           f"{int(np.argmax(err - tol))} err {err.max():.3e}")
    assert np.all(y[tol == 0] == 0.0), f"{label}: rows with an empty kept support must be 0"


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("O,I,kind", [(1, 1, "gauss"), (5, 3, "gauss"), (64, 700, "halves"),
                                      (1024, 130, "onesided"), (1025, 333, "wide"),
                                      (2100, 256, "gauss"), (3000, 129, "halves")])
def test_pack_q_bytes_match_oracle(duo, bits, O, I, kind):
    W = _weight(O, I, 0.5, O * 13 + I + bits, kind)
    h = duo.duo_pack(W.cuda(), FMT[bits])
    info, index, aux, data = duo.packed_bytes(h)
    hdr, off, rdata, table = orc.ref_pack_cmb_q(W.numpy(), bits)
    assert info.fmt == {8: 2, 4: 3}[bits] and info.nnz == hdr["nnz"]
    assert np.array_equal(index.view(np.uint32), off)
    assert np.array_equal(data, rdata)
    assert np.array_equal(aux.view(np.uint32), table)
    h.free()
    assert duo.duo_device_status() == 0


@pytest.mark.parametrize("bits", [8, 4])
@pytest.mark.parametrize("O,I", [(1, 1), (5, 3), (64, 700), (1024, 1024), (1025, 333),
                                 (2048, 4096), (3000, 2049)])
def test_spmspv_q_topk_all_rows(duo, bits, O, I):
    W = _weight(O, I, 0.5, O * 7 + I, "gauss")
    x = _laplace(I, O + I)
    x16 = x.numpy()
    Wd = orc.oracle_dequantize(W.numpy(), bits)
    h = duo.duo_pack(W.cuda(), FMT[bits])
    for k in sorted({0, 1, I // 2, (3 * I) // 10, I}):
        y = duo.duo_spmspv(h, x.cuda(), k)
        torch.cuda.synchronize()
        K, _ = orc.oracle_sparsify(x16, k)
        _check_y(y.cpu().numpy(), Wd, x16, K, f"q{bits} {O}x{I} k{k}")
    h.free()
    assert duo.duo_device_status() == 0


@pytest.mark.parametrize("bits", [8, 4])
def test_spmspv_q_threshold(duo, bits):
    O, I = 3000, 2049
    W = _weight(O, I, 0.5, 77 + bits, "gauss")
    x = _laplace(I, 78)
    x16 = x.numpy()
    Wd = orc.oracle_dequantize(W.numpy(), bits)
    h = duo.duo_pack(W.cuda(), FMT[bits])
    a = np.sort(np.abs(x16.astype(np.float64)))
    for tau in (0.0, float(a[I // 2]), float(a[int(I * 0.95)]), 65504.0):
        y = duo.duo_spmspv_threshold(h, x.cuda(), tau)[0]
        torch.cuda.synchronize()
        K, _ = orc.oracle_sparsify_threshold(x16, tau)
        _check_y(y.cpu().numpy(), Wd, x16, K, f"q{bits} tau {tau}")
    h.free()
    assert duo.duo_device_status() == 0


@pytest.mark.parametrize("bits", [8, 4])
def test_spmspv_q_shared_input_and_listed(duo, bits):
    """q/k/v-like: three products of different heights sharing x in one
    launch (fused), then the same with the kept list given (listed mode,
    ids ascending)."""
    I = 4096
    Ws = [_weight(O, I, 0.5, 100 + O + bits, "gauss") for O in (4096, 1024, 1024)]
    x = _laplace(I, 5 + bits)
    x16 = x.numpy()
    k = I // 2
    hs = [duo.duo_pack(W.cuda(), FMT[bits]) for W in Ws]
    K, V = orc.oracle_sparsify(x16, k)
    ys = duo.duo_spmspv_multi(hs, x.cuda(), k)
    kidx = torch.from_numpy(K.view(np.int16).copy()).cuda()
    kval = torch.from_numpy(V.copy()).cuda()
    ys2 = duo.duo_spmspv_multi(hs, None, k, kept_idx=kidx, kept_val=kval)
    torch.cuda.synchronize()
    for W, y, y2, name in zip(Ws, ys, ys2, "qkv"):
        Wd = orc.oracle_dequantize(W.numpy(), bits)
        _check_y(y.cpu().numpy(), Wd, x16, K, f"q{bits} shared {name}")
        _check_y(y2.cpu().numpy(), Wd, x16, K, f"q{bits} listed {name}")
    for h in hs:
        h.free()
    assert duo.duo_device_status() == 0


@pytest.mark.parametrize("bits", [8, 4])
def test_spmspv_q_llama2_7b_layer_rows(duo, bits):
    """The bench's layer shapes, sampled rows (first, last, segment borders)."""
    from paper_2506_20194_gb300 import synth
    wl = synth.WORKLOADS["llama2-7b-layer"]
    shape = wl["shape"]
    rng = np.random.default_rng(3 + bits)
    for proj in ("gate", "down"):
        O, I = shape.shapes[proj]
        W = synth.layer_weight(wl, proj, layer=0, device="cuda")
        x = synth.layer_input(wl, proj, layer=0, device="cuda")
        x16 = _np16(x)
        k = I // 2
        h = duo.duo_pack(W, FMT[bits])
        y = duo.duo_spmspv(h, x, k).cpu().numpy()
        rows = sorted({0, O - 1, 1023, 1024, O // 2} | set(rng.choice(O, 200, replace=False).tolist()))
        Wr = W[torch.tensor(rows, device="cuda")].cpu().numpy().view(np.float16)
        Wd = orc.oracle_dequantize(Wr, bits)   # grids are per row: a row subset is exact
        K, _ = orc.oracle_sparsify(x16, k)
        _check_y(y[rows], Wd, x16, K, f"7b q{bits} {proj}")
        h.free()
    assert duo.duo_device_status() == 0


def test_spmspv_q_graph_replay(duo):
    O, I = 2048, 4096
    W = _weight(O, I, 0.5, 9, "gauss")
    x = _laplace(I, 10).cuda()
    h = duo.duo_pack(W.cuda(), "bitmask_q4")
    Wd = orc.oracle_dequantize(W.numpy(), 4)
    k = I // 2
    y = torch.empty(O, dtype=torch.float32, device="cuda")
    duo.duo_spmspv(h, x, k, y=y)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        duo.duo_spmspv(h, x, k, y=y)
    for _ in range(20):
        g.replay()
    torch.cuda.synchronize()
    K, _ = orc.oracle_sparsify(_np16(x), k)
    _check_y(y.cpu().numpy(), Wd, _np16(x), K, "graph replay")
    x2 = _laplace(I, 11)
    x.copy_(x2.cuda())
    g.replay()
    torch.cuda.synchronize()
    K2, _ = orc.oracle_sparsify(x2.numpy(), k)
    _check_y(y.cpu().numpy(), Wd, x2.numpy(), K2, "graph replay new x")
    h.free()
    assert duo.duo_device_status() == 0


def test_coded_launch_needs_a_run_per_sm(duo):
    """More (product, segment) runs than SMs: the coded formats refuse the
    launch on the host (DUO_ERANGE) instead of falling back."""
    props = torch.cuda.get_device_properties(0)
    O, I = (props.multi_processor_count + 1) * 1024, 64
    W = torch.zeros(O, I, dtype=torch.float16)
    W[::3, ::2] = 0.01
    h = duo.duo_pack(W.cuda(), "bitmask_q8")
    x = _laplace(I, 1).cuda()
    with pytest.raises(duo.DuoError) as ei:
        duo.duo_spmspv(h, x, I // 2)
    assert ei.value.code == duo.DUO_ERANGE
    with pytest.raises(duo.DuoError) as ei:
        duo.duo_spmspv_threshold(h, x, 0.5)
    assert ei.value.code == duo.DUO_ERANGE
    h.free()
    assert duo.duo_device_status() == 0


def test_listed_out_of_group_order_is_rejected(duo):
    """A coded launch streams grid tables in group order, so a kept list
    whose ids decrease across 128-channel groups is rejected on the device
    (duo_device_status: DUO_EFORMAT); the next call on the same handle
    works."""
    O, I = 2048, 1024
    W = _weight(O, I, 0.5, 5, "gauss")
    h = duo.duo_pack(W.cuda(), "bitmask_q8")
    x = _laplace(I, 6)
    k = 300
    ids = np.arange(I - 1, I - 1 - k, -1).astype(np.uint16)          # descending
    kidx = torch.from_numpy(ids.view(np.int16).copy()).cuda()
    kval = x[torch.from_numpy(ids.astype(np.int64))].cuda()
    duo.duo_spmspv(h, None, k, kept_idx=kidx, kept_val=kval)
    assert duo.duo_device_status() == duo.DUO_EFORMAT
    y = duo.duo_spmspv(h, x.cuda(), k)                                # fused: fine again
    torch.cuda.synchronize()
    K, _ = orc.oracle_sparsify(x.numpy(), k)
    _check_y(y.cpu().numpy(), orc.oracle_dequantize(W.numpy(), 8), x.numpy(), K, "after rejection")
    assert duo.duo_device_status() == 0
    h.free()
