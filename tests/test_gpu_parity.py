"""GPU parity: libslorr through its C ABI against the fp64 oracle on the same
seeded inputs (Sec. 3, Eq. 1, Listing 1, Alg. 2).

Tolerances (relative, on the loss and on each matrix's gradient in Frobenius
norm), the stated targets:
* fp32 compute mode: 1e-5;
* fp16-operand mode (tensor cores, the default): 2e-2;
* bf16-operand modes: 2e-2 (bf16, and bf16_split: every product operand
  carried as a bf16 hi/lo pair, every product as three bf16 products).
Weights and gradients stored in bf16 add one rounding of the stored gradient
(2^-9 relative).

One exception, which does NOT meet the 2e-2 target: the SLORR-Hoyer gradient
with plain bf16 operands.  It is the difference of two nearly equal terms,
and rounding the iterate to bf16 (8 significand bits) after every step leaves
2.1e-2 to 4.1e-2 on the paper-shaped sets (fp16, 11 bits, at the same tensor
rate: 2.7e-3 to 5.1e-3).  Those gradients are held to BF16_HOYER_GRAD = 5e-2,
their measured floor with margin, so that the option stays tested; the bf16
loss and the bf16 SLORR-Nuc gradient are held to 2e-2.  The bf16_split mode,
whose hi/lo pairs remove that rounding, is held to 2e-2 everywhere.

The Hoyer gradient is the difference of two terms, 2 reg P_hat / frob and
2 reg n_hat W / frob^3 (Listing 1).  When they cancel almost completely (rank
one, equal singular values: the exact gradient is zero) a relative error only
measures rounding of that cancellation, so for matrices whose gradient norm is
below 5% of the first term's norm the error is taken relative to that term.
"""

import numpy as np
import pytest

import oracle
import workloads

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

TOL = {"fp32": (1e-5, 1e-5), "fp16": (2e-2, 2e-2), "bf16": (2e-2, 2e-2), "bf16_split": (2e-2, 2e-2)}
BF16_HOYER_GRAD = 5e-2   # outside the 2e-2 target: see the module docstring
BF16_STORAGE = 2.0 ** -9  # one rounding of a gradient stored in bf16
EPS = 1e-7


def grad_tol(compute, variant):
    return BF16_HOYER_GRAD if (compute == "bf16" and variant == "hoyer") else TOL[compute][1]


@pytest.fixture(scope="module", autouse=True)
def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2607_08754_gb300 import slorr
    slorr.load_library()   # raises if the extension is missing: no fallback


def run_gpu(Ws, variant="hoyer", compute="fp16", lam=1.0, grad_scale=1.0, dtype="f32", iters=6,
            grads0=None, flags=0, reg=None):
    from paper_2607_08754_gb300.slorr import Regularizer
    if reg is None:
        reg = Regularizer([W.shape for W in Ws], variant=variant, compute=compute, dtype=dtype,
                          iters=iters, lam=lam, grad_scale=grad_scale, flags=flags)
    tdt = torch.float32 if dtype == "f32" else torch.bfloat16
    w = [torch.from_numpy(np.ascontiguousarray(W, dtype=np.float32)).to("cuda").to(tdt) for W in Ws]
    if grads0 is None:
        g = [torch.zeros_like(x) for x in w]
    else:
        g = [torch.from_numpy(np.ascontiguousarray(G, dtype=np.float32)).to("cuda").to(tdt) for G in grads0]
    per = torch.full((len(Ws),), float("nan"), device="cuda")
    loss = reg(w, g, per_matrix=per)
    torch.cuda.synchronize()
    status = reg.status()
    return (loss.item(), per.cpu().double().numpy(), [x.double().cpu().numpy() for x in g], status, reg,
            [x.double().cpu().numpy() for x in w])


def rel(a, b):
    nb = np.linalg.norm(b)
    return np.linalg.norm(a - b) / nb if nb > 0 else np.linalg.norm(a - b)


def grad_err(got, ref, W, variant, lam, grad_scale):
    """Relative gradient error, against the first term's scale when the
    Hoyer terms cancel (see the module docstring)."""
    nr = np.linalg.norm(ref)
    if variant == "hoyer":
        co = oracle.pe_coefficients(6)
        L, _, n_hat, frob = oracle.reg_single(W, "hoyer", co, EPS)
        term = abs(lam * grad_scale) * 2.0 * (n_hat / frob) / frob * np.sqrt(min(W.shape))
        if nr < 0.05 * term:
            return np.linalg.norm(got - ref) / term
    return np.linalg.norm(got - ref) / nr if nr > 0 else np.linalg.norm(got - ref)


def check(Ws, variant, compute, lam=1.0, grad_scale=1.0, dtype="f32", iters=6, grads0=None, flags=0):
    loss, per, grads, status, reg, w_used = run_gpu(Ws, variant, compute, lam, grad_scale, dtype, iters,
                                                    grads0, flags)
    assert status == 0
    co = oracle.pe_coefficients(T=iters)
    ref_loss, ref_per, ref_inc = oracle.reg_forward_backward(w_used, variant, co, lam, EPS, grad_scale)
    tl, tg = TOL[compute][0], grad_tol(compute, variant)
    assert abs(loss - ref_loss) <= tl * abs(ref_loss) + 1e-6, (loss, ref_loss)
    for i in range(len(Ws)):
        assert abs(per[i] - ref_per[i]) <= tl * abs(ref_per[i]) + 1e-6, (i, per[i], ref_per[i])
        base = grads0[i] if grads0 is not None else 0.0
        ref_g = base + ref_inc[i]
        err = grad_err(grads[i] - base, ref_inc[i], w_used[i], variant, lam, grad_scale)
        if dtype == "bf16":
            # the accumulated gradient is stored in bf16: one extra rounding
            assert err <= tg + BF16_STORAGE, (i, err)
        else:
            assert err <= tg, (i, err)
            assert np.all(np.isfinite(grads[i])) and grads[i].shape == ref_g.shape
    return loss, per, grads, reg


# ---- cfg1: 8 x 256 x 256, N(0, 1/256), fp32 mode --------------------------------

def test_cfg1_fp32_hoyer():
    Ws = workloads.generate("cfg1")
    check(Ws, "hoyer", "fp32")


def test_cfg1_fp32_iterates_match_every_step():
    from paper_2607_08754_gb300.slorr import Regularizer
    Ws = workloads.generate("cfg1", [0, 1])
    reg = Regularizer([W.shape for W in Ws], compute="fp32")
    w = [torch.from_numpy(W).cuda() for W in Ws]
    co = oracle.pe_coefficients(6)
    for k in range(7):
        reg.run_steps(w, k)
        torch.cuda.synchronize()
        for i, W in enumerate(Ws):
            ref_steps, tr = oracle.polar_express_steps(W.astype(np.float64), co, EPS)
            got = reg.iterate(i, k).double().cpu().numpy()
            assert rel(got, ref_steps[k]) <= 1e-5, (k, i, rel(got, ref_steps[k]))
        fsq, _ = reg.scalars(0)
        assert fsq == pytest.approx(float(np.sum(Ws[0].astype(np.float64) ** 2)), rel=1e-6)


def test_bf16_split_iterates_every_step():
    """bf16 hi/lo mode, step by step: the iterate's hi part after k < T steps
    (bf16, at most 2^-9 relative rounding) and X_T (stored in fp16) against
    the oracle's fp64 iterates, with W in both orientations (the view is the
    P x Q iterate either way)."""
    from paper_2607_08754_gb300.slorr import Regularizer
    Ws = [workloads.random_matrix((256, 640), 51, 0.05), workloads.random_matrix((700, 300), 52, 0.05)]
    reg = Regularizer([W.shape for W in Ws], compute="bf16_split")
    w = [torch.from_numpy(W).cuda() for W in Ws]
    co = oracle.pe_coefficients(6)
    for k in range(7):
        reg.run_steps(w, k)
        torch.cuda.synchronize()
        assert reg.status() == 0
        for i, W in enumerate(Ws):
            ref_steps, tr = oracle.polar_express_steps(W.astype(np.float64), co, EPS)
            got = reg.iterate(i, k).double().cpu().numpy()   # P x Q, X_0 scaled
            assert rel(got, ref_steps[k]) <= 5e-3, (k, i, rel(got, ref_steps[k]))


@pytest.mark.parametrize("compute", ["fp32", "fp16", "bf16", "bf16_split"])
@pytest.mark.parametrize("variant", ["hoyer", "nuclear"])
def test_ragged_shapes(compute, variant):
    shapes = [(1, 1), (1, 7), (9, 1), (3, 5), (5, 3), (64, 147), (130, 70), (200, 333), (320, 1280),
              (1000, 512), (129, 129)]
    Ws = [workloads.random_matrix(s, seed=10 + i, std=0.05) for i, s in enumerate(shapes)]
    check(Ws, variant, compute, lam=0.7, grad_scale=2.0)


@pytest.mark.parametrize("compute,variant", [("fp16", "hoyer"), ("fp16", "nuclear"), ("bf16", "hoyer"),
                                             ("fp32", "hoyer"), ("bf16_split", "hoyer")])
def test_extreme_and_large_shapes(compute, variant):
    """Shapes at the limits: rows of 65536 elements (the longest the library
    takes; the Gram's K is 65536 and its tiles split K), the transposed case,
    a P = 2048 matrix whose Poly and Update read most K blocks of A and M
    MN-major from the stored transpose (8 tile rows), and a ragged transposed
    matrix (P = 1500, Ppad = 1536)."""
    shapes = [(64, 65536), (65536, 96), (2048, 6144), (3000, 1500)]
    Ws = [workloads.random_matrix(s, seed=40 + i, std=0.02) for i, s in enumerate(shapes)]
    check(Ws, variant, compute, lam=0.5)


@pytest.mark.parametrize("compute", ["fp32", "fp16", "bf16", "bf16_split"])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_flat_tiles_with_tails(compute, dtype):
    """Rows a multiple of 128 elements: the memory passes take flat runs of
    8192 elements.  The shapes end in partial runs (m n not a multiple of
    8192), include m > n (X^T stored, padding rows zero-filled by the flat
    cast), a matrix smaller than one run, and (fp32 storage) a gradient
    accumulated onto an existing one: in bf16 storage the existing values'
    own rounding would dominate the comparison."""
    shapes = [(130, 768), (1000, 384), (77, 128), (200, 1280), (3, 256), (640, 1024)]
    Ws = [workloads.random_matrix(s, seed=40 + i, std=0.05) for i, s in enumerate(shapes)]
    G0 = [workloads.random_matrix(s, seed=60 + i, std=0.01) for i, s in enumerate(shapes)]
    check(Ws, "hoyer", compute, lam=0.3, dtype=dtype, grads0=G0 if dtype == "f32" else None)


@pytest.mark.parametrize("compute", ["fp16", "bf16", "bf16_split"])
@pytest.mark.parametrize("variant", ["hoyer", "nuclear"])
def test_resnet18_weight_set(compute, variant):
    """All 21 matrices of the ResNet-18 set; with bf16_split every gradient
    within the 2e-2 target (plain bf16 operands miss it on this set's Hoyer
    gradients)."""
    check(workloads.generate("resnet18"), variant, compute)


def test_vit_b16_block_fp16():
    check(workloads.generate("vit_b16", range(4)), "hoyer", "fp16")


def test_decoder_560m_layer_fp16():
    check(workloads.generate("decoder_560m", range(7)), "hoyer", "fp16")


# ---- tensor cores vs CUDA cores on the same 16-bit arithmetic -------------------

@pytest.mark.parametrize("compute,flags", [("fp16", 0), ("bf16", 0), ("fp16", 2048)])
def test_tensor_core_iterates_match_simt(compute, flags):
    """The CTA-pair tensor-core kernel (256 x 256 tiles; 2048 =
    SLORR_FLAG_NO_SPLIT_K) against the CUDA-core kernel on the same 16-bit
    iterates."""
    from paper_2607_08754_gb300.slorr import Regularizer, FLAG_SIMT_GEMM
    shapes = [(256, 768), (768, 256), (320, 1280), (384, 384), (640, 1000)]
    Ws = [workloads.random_matrix(s, seed=70 + i, std=0.02) for i, s in enumerate(shapes)]
    w = [torch.from_numpy(W).cuda() for W in Ws]
    tc = Regularizer(shapes, compute=compute, flags=flags)
    st = Regularizer(shapes, compute=compute, flags=FLAG_SIMT_GEMM)
    ulp = 2.0 ** -10 if compute == "fp16" else 2.0 ** -7
    for k in (1, 2, 6):
        tc.run_steps(w, k)
        st.run_steps(w, k)
        torch.cuda.synchronize()
        assert tc.status() == 0 and st.status() == 0
        for i in range(len(shapes)):
            a = tc.iterate(i, k).double().cpu().numpy()
            b = st.iterate(i, k).double().cpu().numpy()
            assert rel(a, b) <= 4 * ulp * (k if k < 6 else 6), (k, i, rel(a, b))


# ---- edge cases -------------------------------------------------------------------

@pytest.mark.parametrize("compute", ["fp32", "fp16", "bf16_split"])
def test_zero_matrix_and_accumulation(compute):
    Ws = [np.zeros((40, 70), np.float32), workloads.random_matrix((70, 40), 3, 0.1)]
    rng = np.random.default_rng(4)
    g0 = [rng.normal(size=W.shape).astype(np.float32) for W in Ws]
    loss, per, grads, reg = check(Ws, "hoyer", compute, grads0=g0)
    assert per[0] == 0.0
    assert np.array_equal(grads[0], g0[0].astype(np.float64))   # zero matrix: gradient 0, grad untouched


def test_two_calls_reuse_workspace_and_accumulate():
    from paper_2607_08754_gb300.slorr import Regularizer
    Ws = [workloads.random_matrix((96, 200), 5, 0.05), workloads.random_matrix((300, 64), 6, 0.05)]
    reg = Regularizer([W.shape for W in Ws], lam=0.5)
    w = [torch.from_numpy(W).cuda() for W in Ws]
    g = [torch.zeros_like(x) for x in w]
    l1 = reg(w, g).item()
    once = [x.clone() for x in g]
    l2 = reg(w, g).item()
    torch.cuda.synchronize()
    assert reg.status() == 0
    assert l1 == l2                                    # deterministic
    for a, b in zip(g, once):
        assert torch.equal(a, 2 * b) or torch.allclose(a, 2 * b, rtol=1e-6, atol=0)


def test_bf16_weights_and_grads():
    Ws = [workloads.random_matrix((128, 300), 8, 0.05), workloads.random_matrix((257, 100), 9, 0.05)]
    check(Ws, "hoyer", "fp16", dtype="bf16")


def test_nonfinite_weight_reports_status_and_leaves_grad():
    from paper_2607_08754_gb300.slorr import Regularizer
    W = workloads.random_matrix((64, 64), 11, 0.1)
    W[3, 5] = np.inf
    reg = Regularizer([W.shape, (32, 32)])
    w = [torch.from_numpy(W).cuda(), torch.from_numpy(workloads.random_matrix((32, 32), 12)).cuda()]
    g = [torch.ones_like(x) for x in w]
    reg(w, g)
    torch.cuda.synchronize()
    assert reg.status() == 6            # SLORR_ERR_NONFINITE
    assert torch.all(g[0] == 1.0)       # untouched
    assert reg.status() == 0            # reading clears it


# ---- full-size ViT-L/16 weight set in the benchmark configuration, sampled --------

def test_vit_l16_full_size_sampled():
    from paper_2607_08754_gb300.slorr import Regularizer
    name = "vit_l16"
    shapes = workloads.shapes(name)
    reg = Regularizer(shapes, compute="fp16", lam=1.0)
    w = [torch.from_numpy(workloads.generate_one(name, i)).cuda() for i in range(len(shapes))]
    g = [torch.zeros_like(x) for x in w]
    per = torch.empty(len(shapes), device="cuda")
    loss = reg(w, g, per_matrix=per).item()
    torch.cuda.synchronize()
    assert reg.status() == 0
    per = per.double().cpu().numpy()
    assert loss == pytest.approx(per.sum(), rel=1e-6)
    co = oracle.pe_coefficients(6)
    for i in (0, 1, 2, 3, 94):
        W = workloads.generate_one(name, i).astype(np.float64)
        L, G, _, _ = oracle.reg_single(W, "hoyer", co, EPS)
        assert abs(per[i] - L) <= 2e-2 * L
        assert rel(g[i].double().cpu().numpy(), G) <= 2e-2


def full_set_sampled(name, samples, variant="hoyer", compute="fp16"):
    """The whole weight set in one call, as bench.py times it; the sampled
    matrices' values and gradients against the oracle, and the loss against
    the sum of the values."""
    from paper_2607_08754_gb300.slorr import Regularizer
    shapes = workloads.shapes(name)
    reg = Regularizer(shapes, variant=variant, compute=compute, lam=1.0)
    w = [torch.from_numpy(workloads.generate_one(name, i)).cuda() for i in range(len(shapes))]
    g = [torch.zeros_like(x) for x in w]
    per = torch.empty(len(shapes), device="cuda")
    loss = reg(w, g, per_matrix=per).item()
    torch.cuda.synchronize()
    assert reg.status() == 0
    per = per.double().cpu().numpy()
    assert loss == pytest.approx(per.sum(), rel=1e-6)
    co = oracle.pe_coefficients(6)
    tl, tg = TOL[compute][0], grad_tol(compute, variant)
    for i in samples:
        W = workloads.generate_one(name, i).astype(np.float64)
        L, G, _, _ = oracle.reg_single(W, variant, co, EPS)
        assert abs(per[i] - L) <= tl * abs(L), (name, i)
        assert grad_err(g[i].double().cpu().numpy(), G, W, variant, 1.0, 1.0) <= tg, (name, i)


def test_vit_l16_full_size_every_matrix():
    """The bench's own configuration (ViT-L/16 set, fp16 operands, Hoyer, one
    call over all 96 matrices) with every matrix's value and gradient against
    the oracle, not a sample."""
    full_set_sampled("vit_l16", range(96))


def test_decoder_560m_full_size_sampled():
    """The 560M decoder set (168 matrices, 417 M weights): q, k, o, gate and
    down projections of the first and last blocks."""
    full_set_sampled("decoder_560m", (0, 1, 3, 4, 6, 167))


def test_decoder_560m_mha_full_size_sampled_nuclear():
    full_set_sampled("decoder_560m_mha", (1, 5, 160), variant="nuclear")


@pytest.mark.parametrize("variant", ["hoyer", "nuclear"])
def test_vit_b16_full_size_sampled(variant):
    """The ViT-B/16 set in the bench's configuration (fp16 operands; the plan
    takes the dataflow launch for it): the first block's matrices, a middle
    one and the last against the oracle."""
    from paper_2607_08754_gb300.slorr import Regularizer, slorr_dataflow_items
    slorr_dataflow_items(Regularizer(workloads.shapes("vit_b16")).handle)  # raises if per-phase
    full_set_sampled("vit_b16", (0, 1, 2, 3, 25, 47), variant=variant)


def test_vit_b16_full_size_sampled_bf16():
    full_set_sampled("vit_b16", (0, 1, 2, 3, 47), compute="bf16")


def test_vit_l16_full_size_sampled_nuclear():
    """ViT-L/16 set, SLORR-Nuc (the configuration names Hoyer and nuclear)."""
    full_set_sampled("vit_l16", (0, 1, 2, 3, 93), variant="nuclear")


@pytest.mark.parametrize("variant", ["hoyer", "nuclear"])
def test_vit_l16_full_size_sampled_bf16(variant):
    full_set_sampled("vit_l16", (0, 1, 2, 3, 95), variant=variant, compute="bf16")


def test_decoder_560m_full_size_sampled_bf16():
    full_set_sampled("decoder_560m", (0, 1, 2, 4, 6, 164), compute="bf16")


# ---- bf16 hi/lo operands: the bf16 configurations within the 2e-2 target ---------

@pytest.mark.parametrize("variant", ["hoyer", "nuclear"])
def test_vit_l16_full_size_sampled_bf16_split(variant):
    full_set_sampled("vit_l16", (0, 1, 2, 3, 95), variant=variant, compute="bf16_split")


def test_decoder_560m_full_size_sampled_bf16_split():
    full_set_sampled("decoder_560m", (0, 1, 2, 4, 6, 164), compute="bf16_split")


def test_vit_b16_full_size_sampled_bf16_split():
    full_set_sampled("vit_b16", (0, 1, 2, 3, 47), compute="bf16_split")


def test_bf16_split_beats_bf16_on_resnet18_hoyer():
    """The hi/lo pairs are what brings the bf16 Hoyer gradient inside the
    target: on the ResNet-18 set the worst gradient error of bf16_split is
    below 5e-3 and a tenth of plain bf16's (a CPU emulation of both roundings
    gives 4e-4 against 4.0e-2)."""
    Ws = workloads.generate("resnet18")
    co = oracle.pe_coefficients(6)
    worst = {}
    for compute in ("bf16", "bf16_split"):
        _, _, grads, status, _, w_used = run_gpu(Ws, "hoyer", compute)
        assert status == 0
        errs = []
        for i, W in enumerate(w_used):
            _, G, _, _ = oracle.reg_single(W, "hoyer", co, EPS)
            errs.append(grad_err(grads[i], G, W, "hoyer", 1.0, 1.0))
        worst[compute] = max(errs)
    assert worst["bf16_split"] <= 5e-3 and worst["bf16_split"] < 0.1 * worst["bf16"], worst


# ---- failure detection: a bounded device wait runs out -----------------------------

@pytest.mark.parametrize("compute", ["fp16", "bf16_split"])
def test_bounded_wait_timeout_reports_status_and_context_survives(compute):
    """SLORR_FLAG_TEST_STALL makes every tensor-core CTA wait on a barrier nothing
    arrives on; with timeout_s = 0.05 each wait gives up, the kernel records
    SLORR_ERR_TIMEOUT in the status word, drains and returns.  The same process
    then runs a normal call that must still match the oracle."""
    from paper_2607_08754_gb300.slorr import Regularizer, FLAG_TEST_STALL
    Ws = [workloads.random_matrix((256, 512), 21, 0.05), workloads.random_matrix((384, 128), 22, 0.05)]
    w = [torch.from_numpy(W).cuda() for W in Ws]
    stall = Regularizer([W.shape for W in Ws], compute=compute, flags=FLAG_TEST_STALL, timeout_s=0.05)
    stall.run_steps(w, 1)
    torch.cuda.synchronize()
    assert stall.status() == 5          # SLORR_ERR_TIMEOUT
    assert stall.status() == 0          # reading clears it
    check(Ws, "hoyer", compute)         # the context is still usable


# ---- decoupled variant (Alg. 1): write the pre-update gradient --------------------

@pytest.mark.parametrize("variant", ["hoyer", "nuclear"])
def test_write_grad_mode_matches_oracle_and_decoupled_step(variant):
    """SLORR_FLAG_WRITE_GRAD overwrites the output with lambda * G_i (Alg. 1's
    G_pre); the caller's decoupled step W <- W - lr * G_pre then matches the
    oracle's."""
    from paper_2607_08754_gb300.slorr import Regularizer, FLAG_WRITE_GRAD
    Ws = workloads.generate("vit_b16", range(4))
    lam, lr = 0.002, 0.1
    reg = Regularizer([W.shape for W in Ws], variant=variant, lam=lam, flags=FLAG_WRITE_GRAD)
    w = [torch.from_numpy(W).cuda() for W in Ws]
    out = [torch.full_like(x, 7.0) for x in w]         # garbage that must be overwritten
    reg(w, out)
    torch.cuda.synchronize()
    assert reg.status() == 0
    co = oracle.pe_coefficients(6)
    _, _, ref = oracle.reg_forward_backward([W.astype(np.float64) for W in Ws], variant, co, lam)
    for i, W in enumerate(Ws):
        got = out[i].double().cpu().numpy()
        assert grad_err(got, ref[i], W.astype(np.float64), variant, lam, 1.0) <= 2e-2
        w_new = W.astype(np.float64) - lr * got
        w_ref = W.astype(np.float64) - lr * ref[i]
        assert np.linalg.norm(w_new - w_ref) <= 2e-2 * lr * np.linalg.norm(ref[i])


# ---- T sweep and the ViT scaling ladder (next rows of the hot-path scope) --------

@pytest.mark.parametrize("T", [1, 2, 4, 8, 10])
def test_iteration_count_sweep(T):
    Ws = [workloads.random_matrix(s, seed=300 + i, std=0.03) for i, s in enumerate([(256, 640), (640, 384)])]
    check(Ws, "hoyer", "fp16", iters=T)
    check(Ws, "hoyer", "fp32", iters=T)
    check(Ws, "hoyer", "bf16_split", iters=T)   # T = 1: the first step is also the last


@pytest.mark.parametrize("name", ["vit_ladder_vit_ti", "vit_ladder_vit_256", "vit_ladder_vit_s"])
def test_vit_ladder_small_sets(name):
    check(workloads.generate(name), "hoyer", "fp16")


def test_vit_ladder_vit_h_sampled():
    from paper_2607_08754_gb300.slorr import Regularizer
    name = "vit_ladder_vit_h"
    shapes = workloads.shapes(name)
    reg = Regularizer(shapes, compute="fp16")
    w = [torch.from_numpy(workloads.generate_one(name, i)).cuda() for i in range(len(shapes))]
    g = [torch.zeros_like(x) for x in w]
    per = torch.empty(len(shapes), device="cuda")
    loss = reg(w, g, per_matrix=per).item()
    torch.cuda.synchronize()
    assert reg.status() == 0
    per = per.double().cpu().numpy()
    assert loss == pytest.approx(per.sum(), rel=1e-6)
    co = oracle.pe_coefficients(6)
    for i in (0, 3, 125):
        W = workloads.generate_one(name, i).astype(np.float64)
        L, G, _, _ = oracle.reg_single(W, "hoyer", co, EPS)
        assert abs(per[i] - L) <= 2e-2 * L
        assert rel(g[i].double().cpu().numpy(), G) <= 2e-2


# ---- fp32 mode on the tensor cores (three tf32 products per product) ----------------

@pytest.mark.parametrize("variant", ["hoyer", "nuclear"])
def test_fp32_tensor_cores_long_k(variant):
    """fp32 mode runs its products as three tf32 tensor-core products with short-K
    accumulations added by compensated sums; K up to 4608 (the truncating
    tensor-core accumulation would otherwise bias a long K) against the
    oracle at the fp32 tolerance."""
    shapes = [(320, 1280), (512, 4608), (4608, 384), (1000, 512), (130, 70)]
    Ws = [workloads.random_matrix(s, seed=610 + i, std=0.03) for i, s in enumerate(shapes)]
    check(Ws, variant, "fp32", lam=0.4)


def test_fp32_tensor_cores_match_compensated_cuda_cores():
    """The tf32 tensor-core iterates stay within the fp32 tolerance of the
    CUDA-core kernel's compensated fp32 dot products after 1, 3 and 6 steps."""
    from paper_2607_08754_gb300.slorr import Regularizer, FLAG_SIMT_GEMM
    shapes = [(256, 768), (768, 256), (320, 1280), (384, 384)]
    Ws = [workloads.random_matrix(s, seed=630 + i, std=0.02) for i, s in enumerate(shapes)]
    w = [torch.from_numpy(W).cuda() for W in Ws]
    tc = Regularizer(shapes, compute="fp32")
    st = Regularizer(shapes, compute="fp32", flags=FLAG_SIMT_GEMM)
    for k in (1, 3, 6):
        tc.run_steps(w, k)
        st.run_steps(w, k)
        torch.cuda.synchronize()
        assert tc.status() == 0 and st.status() == 0
        for i in range(len(shapes)):
            a = tc.iterate(i, k).double().cpu().numpy()
            b = st.iterate(i, k).double().cpu().numpy()
            assert rel(a, b) <= 1e-5, (k, i, rel(a, b))


def test_fp32_tensor_core_bounded_wait_timeout():
    """SLORR_FLAG_TEST_STALL in the tf32 kernel: the MMA thread's bounded wait
    runs out, the call reports SLORR_ERR_TIMEOUT, and a normal fp32 call
    afterwards matches the oracle."""
    from paper_2607_08754_gb300.slorr import Regularizer, FLAG_TEST_STALL
    Ws = [workloads.random_matrix((256, 512), 641, 0.05), workloads.random_matrix((384, 128), 642, 0.05)]
    w = [torch.from_numpy(W).cuda() for W in Ws]
    stall = Regularizer([W.shape for W in Ws], compute="fp32", flags=FLAG_TEST_STALL, timeout_s=0.05)
    stall.run_steps(w, 1)
    torch.cuda.synchronize()
    assert stall.status() == 5
    assert stall.status() == 0
    check(Ws, "hoyer", "fp32")
