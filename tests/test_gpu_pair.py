"""The CTA-pair tensor-core kernel (tcgen05 cta_group::2, 256 x 256 tiles over
two SMs, two accumulators per SM) against the CUDA-core path and the oracle.

Shapes are chosen to reach every tile case of the pair kernel: a last row tile
with only 128 rows (the odd CTA's half idle), last column tiles of 128 columns
(64 B rows per CTA), K-major and MN-major operands (m <= n and m > n), a
matrix smaller than one tile, and more tiles than pairs.

Tolerances are those of the tensor-core-vs-CUDA-core test: 4 ulp of the
operand type per step (at most 6 steps' worth), and the oracle parity bounds
(2e-2 for fp16 operands)."""

import numpy as np
import pytest

import oracle
import workloads

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

EPS = 1e-7
SHAPES = [(256, 768), (768, 256), (320, 1280), (384, 384), (640, 1000), (64, 64), (130, 700), (1000, 130)]


@pytest.fixture(scope="module", autouse=True)
def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2607_08754_gb300 import slorr
    slorr.load_library()


def rel(a, b):
    return np.linalg.norm(a - b) / np.linalg.norm(b)


@pytest.mark.parametrize("compute", ["fp16", "bf16"])
def test_pair_iterates_match_simt(compute):
    from paper_2607_08754_gb300.slorr import Regularizer, FLAG_SIMT_GEMM
    Ws = [workloads.random_matrix(s, seed=90 + i, std=0.02) for i, s in enumerate(SHAPES)]
    w = [torch.from_numpy(W).cuda() for W in Ws]
    tc = Regularizer(SHAPES, compute=compute)
    st = Regularizer(SHAPES, compute=compute, flags=FLAG_SIMT_GEMM)
    ulp = 2.0 ** -10 if compute == "fp16" else 2.0 ** -7
    for k in (1, 2, 6):
        tc.run_steps(w, k)
        st.run_steps(w, k)
        torch.cuda.synchronize()
        assert tc.status() == 0 and st.status() == 0
        for i in range(len(SHAPES)):
            a = tc.iterate(i, k).double().cpu().numpy()
            b = st.iterate(i, k).double().cpu().numpy()
            assert rel(a, b) <= 4 * ulp * (k if k < 6 else 6), (k, i, SHAPES[i], rel(a, b))


@pytest.mark.parametrize("variant", ["hoyer", "nuclear"])
def test_pair_forward_backward_matches_oracle(variant):
    from paper_2607_08754_gb300.slorr import Regularizer
    Ws = [workloads.random_matrix(s, seed=120 + i, std=0.05) for i, s in enumerate(SHAPES)]
    Ws += workloads.generate("resnet18", [0, 5, 12, 20])
    shapes = [W.shape for W in Ws]
    reg = Regularizer(shapes, variant=variant, compute="fp16", lam=0.5)
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


def test_pair_vit_l16_layers_match_simt():
    """Paper-sized matrices (one ViT-L/16 block): the pair kernel and the
    CUDA-core kernel give the same iterates up to 16-bit rounding."""
    from paper_2607_08754_gb300.slorr import Regularizer, FLAG_SIMT_GEMM
    Ws = workloads.generate("vit_l16", [0, 1, 2, 3])
    shapes = [W.shape for W in Ws]
    w = [torch.from_numpy(W).cuda() for W in Ws]
    a_reg = Regularizer(shapes)
    b_reg = Regularizer(shapes, flags=FLAG_SIMT_GEMM)
    a_reg.run_steps(w, 6)
    b_reg.run_steps(w, 6)
    torch.cuda.synchronize()
    assert a_reg.status() == 0 and b_reg.status() == 0
    for i in range(len(shapes)):
        a = a_reg.iterate(i, 6).double().cpu().numpy()
        b = b_reg.iterate(i, 6).double().cpu().numpy()
        assert rel(a, b) <= 24 * 2.0 ** -10, (i, rel(a, b))


@pytest.mark.parametrize("mode", ["dataflow", "phase_launches"])
def test_pair_bounded_wait_timeout_and_recovery(mode):
    """SLORR_FLAG_TEST_STALL in the pair kernel: the even CTA's MMA thread waits on
    a barrier nothing arrives on, gives up after timeout_s, and sets both CTAs'
    abort flags; every role unwinds, the even CTA drains the pair's copies, and
    the call reports SLORR_ERR_TIMEOUT.  In the dataflow launch the other pairs'
    producers, waiting for completions that never come, see the timeout in the
    status word and unwind too.  A normal pair call afterwards matches the
    CUDA-core path."""
    from paper_2607_08754_gb300.slorr import (Regularizer, FLAG_TEST_STALL, FLAG_SIMT_GEMM, FLAG_PHASE_LAUNCHES,
                                              FLAG_DATAFLOW)
    shapes = [(256, 512), (384, 128), (640, 1000)]
    Ws = [workloads.random_matrix(s, 31 + i, 0.05) for i, s in enumerate(shapes)]
    w = [torch.from_numpy(W).cuda() for W in Ws]
    extra = FLAG_PHASE_LAUNCHES if mode == "phase_launches" else FLAG_DATAFLOW
    stall = Regularizer(shapes, flags=FLAG_TEST_STALL | extra, timeout_s=0.05)
    stall.run_steps(w, 1)
    torch.cuda.synchronize()
    assert stall.status() == 5          # SLORR_ERR_TIMEOUT
    assert stall.status() == 0
    tc = Regularizer(shapes, flags=extra)
    st = Regularizer(shapes, flags=FLAG_SIMT_GEMM)
    tc.run_steps(w, 2)
    st.run_steps(w, 2)
    torch.cuda.synchronize()
    assert tc.status() == 0 and st.status() == 0
    for i in range(len(shapes)):
        a = tc.iterate(i, 2).double().cpu().numpy()
        b = st.iterate(i, 2).double().cpu().numpy()
        assert rel(a, b) <= 8 * 2.0 ** -10, (i, rel(a, b))


def test_programmatic_dependent_launch_is_bit_identical():
    """Programmatic dependent launch (the default; SLORR_FLAG_NO_PDL turns it
    off) only changes when kernels launch, not what they compute: three
    consecutive calls (accumulating into .grad) and the loss equal the
    serialised launches bit for bit."""
    from paper_2607_08754_gb300.slorr import Regularizer, FLAG_NO_PDL
    Ws = [workloads.random_matrix(s, seed=900 + i, std=0.05) for i, s in enumerate(SHAPES)]
    out = []
    for flags in (0, FLAG_NO_PDL):
        reg = Regularizer(SHAPES, flags=flags)
        w = [torch.from_numpy(W).cuda() for W in Ws]
        g = [torch.zeros_like(x) for x in w]
        losses = [reg(w, g).clone() for _ in range(3)]
        torch.cuda.synchronize()
        assert reg.status() == 0
        out.append(([x.cpu() for x in g], torch.cat(losses).cpu()))
    for a, b in zip(out[0][0], out[1][0]):
        assert torch.equal(a, b)
    assert torch.equal(out[0][1], out[1][1])


def test_split_k_gram_matches_whole_k_and_oracle():
    """Split K of long Gram tiles (the default for sets whose few Gram tiles
    have a long K): the parts' fp32 partials, added in part order by the last
    part's epilogue, give the same iterates as whole-K tiles
    (SLORR_FLAG_NO_SPLIT_K) up to fp32 summation order, and the values and
    gradients match the oracle.  Shapes: K = Q up to 4608, a transposed
    matrix (m > n: MN-major Gram operands), a tile of 128 rows and a set
    small enough that its tiles are split."""
    from paper_2607_08754_gb300.slorr import Regularizer, FLAG_NO_SPLIT_K, slorr_gemm_items
    shapes = [(512, 4608), (4608, 384), (256, 2304), (130, 1152), (512, 1000)]
    Ws = [workloads.random_matrix(s, seed=510 + i, std=0.02) for i, s in enumerate(shapes)]
    w = [torch.from_numpy(W).cuda() for W in Ws]
    split = Regularizer(shapes)
    whole = Regularizer(shapes, flags=FLAG_NO_SPLIT_K)
    assert slorr_gemm_items(split.handle, 0) > slorr_gemm_items(whole.handle, 0)
    for k in (1, 2, 6):
        split.run_steps(w, k)
        whole.run_steps(w, k)
        torch.cuda.synchronize()
        assert split.status() == 0 and whole.status() == 0
        for i in range(len(shapes)):
            a = split.iterate(i, k).double().cpu().numpy()
            b = whole.iterate(i, k).double().cpu().numpy()
            assert rel(a, b) <= 4 * 2.0 ** -10 * k, (k, i, shapes[i], rel(a, b))
    g = [torch.zeros_like(x) for x in w]
    per = torch.empty(len(shapes), device="cuda")
    loss = split(w, g, per_matrix=per).item()
    torch.cuda.synchronize()
    assert split.status() == 0
    co = oracle.pe_coefficients(6)
    ref_loss, ref_per, ref_inc = oracle.reg_forward_backward([W.astype(np.float64) for W in Ws], "hoyer", co,
                                                             1.0, EPS)
    assert abs(loss - ref_loss) <= 2e-2 * abs(ref_loss)
    per = per.double().cpu().numpy()
    for i in range(len(shapes)):
        assert abs(per[i] - ref_per[i]) <= 2e-2 * abs(ref_per[i]), (i, shapes[i])
        assert rel(g[i].double().cpu().numpy(), ref_inc[i]) <= 2e-2, (i, shapes[i])


def test_split_k_is_deterministic():
    """The last part adds every part's partial in part order, so repeated
    calls give bit-identical iterates whichever part finishes last."""
    from paper_2607_08754_gb300.slorr import Regularizer
    shapes = [(512, 4608), (256, 2304), (512, 1000)]
    Ws = [workloads.random_matrix(s, seed=530 + i, std=0.02) for i, s in enumerate(shapes)]
    w = [torch.from_numpy(W).cuda() for W in Ws]
    reg = Regularizer(shapes)
    outs = []
    for _ in range(3):
        reg.run_steps(w, 6)
        torch.cuda.synchronize()
        assert reg.status() == 0
        outs.append([reg.iterate(i, 6).cpu() for i in range(len(shapes))])
    for o in outs[1:]:
        for a, b in zip(outs[0], o):
            assert torch.equal(a, b)


@pytest.mark.parametrize("compute", ["fp16", "bf16"])
def test_dataflow_launch_is_bit_identical_to_phase_launches(compute):
    """The dataflow launch (every Gram, Poly and Update tile of the T steps in
    one launch, ordered by per-matrix completion counts) computes
    each tile exactly as the per-phase launches (SLORR_FLAG_PHASE_LAUNCHES)
    do: the same K order, split-K parts and epilogue arithmetic.  Iterates
    after 1, 2 and 6 steps (slorr_run_steps skips the later steps' items of
    the dataflow plan), per-matrix values, gradients and the loss are equal
    bit for bit, on a set with every tile case and split-K Gram tiles."""
    from paper_2607_08754_gb300.slorr import Regularizer, FLAG_PHASE_LAUNCHES, FLAG_DATAFLOW, slorr_gemm_item_list
    Ws = [workloads.random_matrix(s, seed=800 + i, std=0.02) for i, s in enumerate(SHAPES)]
    Ws += [workloads.random_matrix(s, seed=820 + i, std=0.02) for i, s in enumerate([(512, 4608), (4608, 384)])]
    Ws += workloads.generate("resnet18", [0, 7, 15, 20])
    shapes = [W.shape for W in Ws]
    w = [torch.from_numpy(W).cuda() for W in Ws]
    df = Regularizer(shapes, compute=compute, flags=FLAG_DATAFLOW)
    ph = Regularizer(shapes, compute=compute, flags=FLAG_PHASE_LAUNCHES)
    assert (slorr_gemm_item_list(df.handle, 0)[:, 6] > 1).any()   # some Gram tiles are split
    for k in (1, 2, 6):
        df.run_steps(w, k)
        ph.run_steps(w, k)
        torch.cuda.synchronize()
        assert df.status() == 0 and ph.status() == 0
        for i in range(len(shapes)):
            assert torch.equal(df.iterate(i, k).cpu(), ph.iterate(i, k).cpu()), (k, i, shapes[i])
    out = []
    for reg in (df, ph):
        g = [torch.zeros_like(x) for x in w]
        per = torch.empty(len(shapes), device="cuda")
        loss = reg(w, g, per_matrix=per)
        torch.cuda.synchronize()
        assert reg.status() == 0
        out.append((loss.cpu(), per.cpu(), [x.cpu() for x in g]))
    assert torch.equal(out[0][0], out[1][0]) and torch.equal(out[0][1], out[1][1])
    for a, b in zip(out[0][2], out[1][2]):
        assert torch.equal(a, b)
