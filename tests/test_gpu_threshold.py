"""GPU parity of the threshold-mask path (§5, threshold-based activation
sparsity) through the C ABI against the CPU oracle.

Bar: kept channel ids / values bit-exact; y within 2e-3 * sum_{j in K}
|W_ij| |x_j| per row, and exactly 0 where that sum is 0.
"""
import numpy as np
import pytest
import torch

import oracle as orc

pytestmark = pytest.mark.gpu

REL_TOL = 2e-3


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


def _weight(O, I, pw, seed):
    g = torch.Generator().manual_seed(seed)
    W = (torch.randn(O, I, generator=g) * 0.02).to(torch.float16)
    W[torch.rand(O, I, generator=g) < pw] = 0
    return W


def _check_y(y_gpu, W16, x16, tau, label):
    K, _ = orc.oracle_sparsify_threshold(x16, tau)
    y_ref = orc.oracle_spmspv_threshold(W16, x16, tau)
    tol = orc.tolerance_rows(W16, x16, K, REL_TOL)
    y = np.asarray(y_gpu, dtype=np.float64)
    err = np.abs(y - y_ref)
    bad = err > tol
    assert not bad.any(), (f"{label}: {bad.sum()} rows out of tolerance; worst row "
                           f"{int(np.argmax(err - tol))} err {err.max():.3e}")
    assert np.all(y[tol == 0] == 0.0), f"{label}: rows with an empty kept support must be 0"


def _median_tau(x16):
    a = np.sort(np.abs(x16.astype(np.float64)))
    return float(a[len(a) // 2])


@pytest.mark.parametrize("I", [1, 31, 32, 33, 1000, 4096, 11008, 28672, 65535])
def test_sparsify_threshold_bit_exact(duo, I):
    xs = {"laplace": _laplace(I, I),
          "ties": (torch.randint(-3, 4, (I,), generator=torch.Generator().manual_seed(I)).to(torch.float16) * 0.5),
          "zeros": torch.zeros(I, dtype=torch.float16)}
    for name, x in xs.items():
        x16 = x.numpy()
        for tau in (0.0, 0.5, _median_tau(x16), 1.0, 65504.0):
            idx, val, cnt = duo.duo_sparsify_threshold(x.cuda(), tau)
            torch.cuda.synchronize()
            n = int(cnt.item())
            K, V = orc.oracle_sparsify_threshold(x16, tau)
            assert n == len(K), (name, I, tau)
            assert np.array_equal(idx[:n].cpu().numpy().view(np.uint16), K), (name, I, tau)
            assert np.array_equal(val[:n].cpu().numpy().view(np.uint16), V.view(np.uint16))
    assert duo.duo_device_status() == 0


@pytest.mark.parametrize("O,I", [(1, 1), (5, 3), (64, 700), (1024, 1024), (1025, 333), (2048, 4096),
                                 (3000, 2049)])
def test_spmspv_threshold_all_rows(duo, O, I):
    W = _weight(O, I, 0.5, O * 7 + I)
    x = _laplace(I, O + I)
    x16 = x.numpy()
    h = duo.duo_pack(W.cuda(), "bitmask")
    for tau in (0.0, _median_tau(x16), 2.0, 65504.0):
        y = duo.duo_spmspv_threshold(h, x.cuda(), tau)[0]
        torch.cuda.synchronize()
        _check_y(y.cpu().numpy(), W.numpy(), x16, tau, f"{O}x{I} tau{tau}")
    h.free()
    assert duo.duo_device_status() == 0


def test_spmspv_threshold_shared_input(duo):
    """q/k/v-like: three products of different heights sharing x in one launch."""
    I = 4096
    Ws = [_weight(O, I, 0.5, 100 + O) for O in (4096, 1024, 1024)]
    x = _laplace(I, 5)
    x16 = x.numpy()
    hs = [duo.duo_pack(W.cuda(), "bitmask") for W in Ws]
    tau = _median_tau(x16)
    ys = duo.duo_spmspv_threshold(hs, x.cuda(), tau)
    torch.cuda.synchronize()
    for W, y, name in zip(Ws, ys, "qkv"):
        _check_y(y.cpu().numpy(), W.numpy(), x16, tau, f"shared {name}")
    for h in hs:
        h.free()


def test_spmspv_threshold_llama2_7b_layer_rows(duo):
    """The bench's layer shapes, sampled rows (first, last, segment borders)."""
    from paper_2506_20194_gb300 import synth
    wl = synth.WORKLOADS["llama2-7b-layer"]
    shape = wl["shape"]
    rng = np.random.default_rng(3)
    for proj in ("gate", "down"):
        O, I = shape.shapes[proj]
        W = synth.layer_weight(wl, proj, layer=0, device="cuda")
        x = synth.layer_input(wl, proj, layer=0, device="cuda")
        x16 = _np16(x)
        tau = _median_tau(x16)
        h = duo.duo_pack(W, "bitmask")
        y = duo.duo_spmspv_threshold(h, x, tau)[0].cpu().numpy()
        rows = sorted({0, O - 1, 1023, 1024, O // 2} | set(rng.choice(O, 200, replace=False).tolist()))
        Wr = W[torch.tensor(rows, device="cuda")].cpu().numpy().view(np.float16)
        _check_y(y[rows], Wr, x16, tau, f"7b {proj}")
        h.free()
    assert duo.duo_device_status() == 0


def test_spmspv_threshold_graph_replay(duo):
    O, I = 2048, 4096
    W = _weight(O, I, 0.5, 9)
    x = _laplace(I, 10).cuda()
    h = duo.duo_pack(W.cuda(), "bitmask")
    tau = _median_tau(_np16(x))
    y = torch.empty(O, dtype=torch.float32, device="cuda")
    duo.duo_spmspv_threshold(h, x, tau, ys=[y])
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        duo.duo_spmspv_threshold(h, x, tau, ys=[y])
    for _ in range(20):
        g.replay()
    torch.cuda.synchronize()
    _check_y(y.cpu().numpy(), W.numpy(), _np16(x), tau, "graph replay")
    x2 = _laplace(I, 11)
    x.copy_(x2.cuda())
    g.replay()
    torch.cuda.synchronize()
    _check_y(y.cpu().numpy(), W.numpy(), x2.numpy(), tau, "graph replay new x")
    h.free()
    assert duo.duo_device_status() == 0
