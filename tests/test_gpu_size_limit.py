"""Matrices at the C ABI's size limit: rows x cols just under 2^31 elements.

Two elongated shapes, 1024 x 2097144 and its transpose (2^31 - 8192
elements each), one MALT step each with bf16 W and fp32 state, and one
MALTER step of the tall one (its prescale also re-reads G for ||L G R||).
Element offsets reach 2^31 - 8, byte offsets of the fp32 buffers 2^33; the Gram
product reduces over 2,097,144 columns; the tall matrix runs every
transposed path (prescale through shared memory, O stored in W's layout).
The fp64 oracle would take hours at this size, so the step is checked
through properties that hold at any size, computed on the host from the
step's inputs and its own intermediates:

* momentum: M = fl32((1 - mu1) G) bitwise (M starts at zero; Algorithm 1,
  M_t line);
* statistics: l = (1 - mu2) rowsum(G^2), r = (1 - mu2) colsum(G^2) within
  1e-5 (Algorithm 1, l_t and r_t lines), every entry;
* preconditioners: L = (l + eps)^(-1/8), R = (r + eps)^(-1/8) within 1e-5,
  every entry;
* graft: ||O||_F and ||L O R||_F from the last GEMM epilogue's partial sums
  within 1e-4 of fp64 norms of the step's O, L, R;
* Newton-Schulz output: finite, with mean squared singular value
  ||O||_F^2 / min(rows, cols) inside the band of the quintic;
* MALTER: ||L G R||^2 within 1e-4 of the fp64 sum over the step's L, R and
  G, nu = (1 - mu2) ||L G R||^2 and alpha = 1 at t = 1 (Algorithm 2, nu_t
  and alpha_t lines);
* update: on sampled rows (the first, the last and random ones) the stored
  bf16 W is the round-to-nearest-even of W_prev - s L O R, s the step's
  scale, wherever no rounding boundary lies within the kernel's fp32 slack
  (Algorithm 1, W_t line).
"""
import numpy as np
import pytest

from tests.gpu_harness import bf16_rounding

pytestmark = pytest.mark.gpu

LIMIT_SHAPES = [(1024, 2097144), (2097144, 1024)]
CHUNK = 1 << 25            # elements per host chunk


def _row_chunks(rows, cols):
    step = max(1, CHUNK // cols)
    for r0 in range(0, rows, step):
        yield r0, min(rows, r0 + step)


@pytest.mark.parametrize("rows,cols,malter", [(r, c, False) for r, c in LIMIT_SHAPES] +
                         [(LIMIT_SHAPES[1][0], LIMIT_SHAPES[1][1], True)])
def test_size_limit(rows, cols, malter):
    import torch
    import paper_2608_05088_gb300.malt as malt
    assert rows * cols < 2 ** 31 and rows * cols > 2 ** 31 - 2 ** 14
    dev = torch.device("cuda:0")
    gen = torch.Generator(device=dev)
    gen.manual_seed(20260 + rows)
    G = torch.empty((rows, cols), dtype=torch.float32, device=dev)
    W = torch.empty((rows, cols), dtype=torch.bfloat16, device=dev)
    for r0, r1 in _row_chunks(rows, cols):
        G[r0:r1].normal_(generator=gen)
        W[r0:r1] = (0.02 * torch.randn((r1 - r0, cols), generator=gen, device=dev)).to(torch.bfloat16)
    M = torch.empty((rows, cols), dtype=torch.float32, device=dev)
    l = torch.empty(rows, dtype=torch.float32, device=dev)
    r = torch.empty(cols, dtype=torch.float32, device=dev)
    W_prev = W.clone()
    opt = malt.MaltOptimizer([(W, G, M, l, r)])
    hp = malt.hparams(lr=0.02)
    opt.step(hp, malter=malter)
    assert opt.check() == malt.MALT_OK
    torch.cuda.synchronize()

    mu1, mu2, eps = np.float32(hp.mu1), np.float32(hp.mu2), np.float32(hp.eps)
    om1 = torch.tensor(np.float32(1) - mu1)
    rs = torch.zeros(rows, dtype=torch.float64)
    cs = torch.zeros(cols, dtype=torch.float64)
    for r0, r1 in _row_chunks(rows, cols):
        g = G[r0:r1].cpu()
        assert torch.equal(M[r0:r1].cpu(), g * om1), (r0, r1)
        g64 = g.double()
        rs[r0:r1] = (g64 * g64).sum(dim=1)
        cs += (g64 * g64).sum(dim=0)
    l_ref = (1.0 - float(mu2)) * rs.numpy()
    r_ref = (1.0 - float(mu2)) * cs.numpy()
    l_gpu = l.cpu().double().numpy()
    r_gpu = r.cpu().double().numpy()
    assert np.max(np.abs(l_gpu - l_ref) / l_ref) < 1e-5
    assert np.max(np.abs(r_gpu - r_ref) / r_ref) < 1e-5
    L, R = (t.cpu().double() for t in opt.precond(0))
    assert np.max(np.abs(L.numpy() - (l_ref + float(eps)) ** -0.125) / L.numpy()) < 1e-5
    assert np.max(np.abs(R.numpy() - (r_ref + float(eps)) ** -0.125) / R.numpy()) < 1e-5

    O = opt.direction(0)
    torch.cuda.synchronize()
    so = 0.0
    sd = 0.0
    slgr = 0.0
    for r0, r1 in _row_chunks(rows, cols):
        o = O[r0:r1].cpu().double()
        assert bool(torch.isfinite(o).all()), (r0, r1)
        d = L[r0:r1, None] * o * R[None, :]
        so += float((o * o).sum())
        sd += float((d * d).sum())
        if malter:
            lgr = L[r0:r1, None] * G[r0:r1].cpu().double() * R[None, :]
            slgr += float((lgr * lgr).sum())
    nO, nD = np.sqrt(so), np.sqrt(sd)
    sc = opt.debug_scalars()[0]
    assert abs(sc[0] - nO) / nO < 1e-4 and abs(sc[1] - nD) / nD < 1e-4, (sc[:2], nO, nD)
    if malter:
        # Algorithm 2 at t = 1 from zero state: nu = (1 - mu2) ||L G R||^2, and
        # alpha = sqrt(1 - mu2) ||Mt|| / ((1 - mu1 + eps)(sqrt(nu) + eps)) with
        # Mt = (1 - mu1) L G R, i.e. 1 up to eps terms
        assert abs(sc[3] - slgr) / slgr < 1e-4, (sc[3], slgr)
        assert abs(sc[4] - (1.0 - float(mu2)) * slgr) / ((1.0 - float(mu2)) * slgr) < 1e-4
        assert abs(sc[5] - 1.0) < 1e-4, sc[5]
    # 5 quintic iterations leave every normalised singular value of a
    # full-rank input in roughly [0.68, 1.2] (bf16 adds a few percent)
    assert 0.4 < so / min(rows, cols) < 1.5, so / min(rows, cols)

    rng = np.random.default_rng(rows)
    want = max(1, (1 << 24) // cols)                  # about 16 M sampled elements
    sample = np.unique(np.concatenate([[0, rows - 1], rng.integers(0, rows, size=want)]))
    idx = torch.from_numpy(sample).to(dev)
    o = O.index_select(0, idx).cpu().double().numpy()
    w_new = W.index_select(0, idx).cpu().double().numpy()
    w_old = W_prev.index_select(0, idx).cpu().double().numpy()
    dW = float(sc[6]) * L.numpy()[sample, None] * o * R.numpy()[None, :]
    w_pre = w_old - dW
    e = bf16_rounding(w_new, w_pre, w_pre, 2.0 ** -21 * (np.abs(w_pre) + np.abs(dW)), dW)
    assert e["own_mismatch"] == 0, e
    assert opt.guard_bytes_corrupted() == 0
