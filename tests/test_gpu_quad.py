"""The 4-CTA kernel (SLORR_FLAG_TC_QUAD: two CTA pairs per cluster computing two
tiles that share an operand, loaded once by TMA multicast) against the
CUDA-core path, the pair kernel and the oracle.

The shapes produce every kind of super-tile: two tiles of one row (shared A
rows), two leftovers of one column (shared B columns), a lone leftover (the
second pair idle), last row tiles of 128 rows and last column tiles of 128
columns, K-major and MN-major operands.  Tolerances as in test_gpu_pair.py."""

import numpy as np
import pytest

import oracle
import workloads

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

EPS = 1e-7
QUAD = 256   # SLORR_FLAG_TC_QUAD
SHAPES = [(256, 768), (768, 256), (320, 1280), (384, 384), (640, 1000), (64, 64), (130, 700), (1000, 130),
          (768, 3072)]


@pytest.fixture(scope="module", autouse=True)
def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2607_08754_gb300 import slorr
    slorr.load_library()


def rel(a, b):
    return np.linalg.norm(a - b) / np.linalg.norm(b)


@pytest.mark.parametrize("compute", ["fp16", "bf16"])
def test_quad_iterates_match_simt_and_pair(compute):
    from paper_2607_08754_gb300.slorr import Regularizer, FLAG_SIMT_GEMM, FLAG_NO_SPLIT_K
    Ws = [workloads.random_matrix(s, seed=500 + i, std=0.02) for i, s in enumerate(SHAPES)]
    w = [torch.from_numpy(W).cuda() for W in Ws]
    qd = Regularizer(SHAPES, compute=compute, flags=QUAD)
    pr = Regularizer(SHAPES, compute=compute, flags=FLAG_NO_SPLIT_K)  # the quad kernel takes whole-K tiles
    st = Regularizer(SHAPES, compute=compute, flags=FLAG_SIMT_GEMM)
    ulp = 2.0 ** -10 if compute == "fp16" else 2.0 ** -7
    for k in (1, 2, 6):
        for r in (qd, pr, st):
            r.run_steps(w, k)
        torch.cuda.synchronize()
        assert qd.status() == 0 and pr.status() == 0 and st.status() == 0
        for i in range(len(SHAPES)):
            a = qd.iterate(i, k).double().cpu().numpy()
            b = st.iterate(i, k).double().cpu().numpy()
            c = pr.iterate(i, k).double().cpu().numpy()
            assert rel(a, b) <= 4 * ulp * (k if k < 6 else 6), (k, i, SHAPES[i], rel(a, b))
            # same tiles, same K order: the quad and pair kernels agree exactly.  The pair
            # kernel stages its epilogue chunks in shared memory and the quad kernel stores
            # them directly, so this also checks the staging (rows, transposed iterates,
            # mirrored blocks, Poly's b A)
            assert np.array_equal(a, c), (k, i, SHAPES[i], rel(a, c))


@pytest.mark.parametrize("variant", ["hoyer", "nuclear"])
def test_quad_forward_backward_matches_oracle(variant):
    from paper_2607_08754_gb300.slorr import Regularizer
    Ws = [workloads.random_matrix(s, seed=600 + i, std=0.05) for i, s in enumerate(SHAPES)]
    Ws += workloads.generate("resnet18", [0, 5, 12, 20])
    shapes = [W.shape for W in Ws]
    reg = Regularizer(shapes, variant=variant, compute="fp16", lam=0.5, flags=QUAD)
    w = [torch.from_numpy(W).cuda() for W in Ws]
    g = [torch.zeros_like(x) for x in w]
    per = torch.empty(len(Ws), device="cuda")
    loss = reg(w, g, per_matrix=per).item()
    torch.cuda.synchronize()
    assert reg.status() == 0
    co = oracle.pe_coefficients(6)
    ref_loss, ref_per, ref_inc = oracle.reg_forward_backward([W.astype(np.float64) for W in Ws], variant, co,
                                                             0.5, EPS)
    assert abs(loss - ref_loss) <= 2e-2 * abs(ref_loss)
    per = per.double().cpu().numpy()
    for i in range(len(Ws)):
        assert abs(per[i] - ref_per[i]) <= 2e-2 * abs(ref_per[i]), (i, shapes[i])
        assert rel(g[i].double().cpu().numpy(), ref_inc[i]) <= 2e-2, (i, shapes[i])


def test_quad_bounded_wait_timeout_and_recovery():
    """SLORR_FLAG_TEST_STALL: both pair leaders' MMA threads wait on a barrier
    nothing arrives on and give up after timeout_s; all four CTAs unwind, each
    leader drains its pair's copies, and the call reports SLORR_ERR_TIMEOUT.  A
    normal call afterwards matches the pair kernel."""
    from paper_2607_08754_gb300.slorr import Regularizer, FLAG_TEST_STALL, FLAG_NO_SPLIT_K
    shapes = [(256, 512), (384, 128), (640, 1000)]
    Ws = [workloads.random_matrix(s, 41 + i, 0.05) for i, s in enumerate(shapes)]
    w = [torch.from_numpy(W).cuda() for W in Ws]
    stall = Regularizer(shapes, flags=QUAD | FLAG_TEST_STALL, timeout_s=0.05)
    stall.run_steps(w, 1)
    torch.cuda.synchronize()
    assert stall.status() == 5          # SLORR_ERR_TIMEOUT
    assert stall.status() == 0
    qd = Regularizer(shapes, flags=QUAD)
    pr = Regularizer(shapes, flags=FLAG_NO_SPLIT_K)
    qd.run_steps(w, 2)
    pr.run_steps(w, 2)
    torch.cuda.synchronize()
    assert qd.status() == 0 and pr.status() == 0
    for i in range(len(shapes)):
        assert np.array_equal(qd.iterate(i, 2).cpu().numpy(), pr.iterate(i, 2).cpu().numpy())
