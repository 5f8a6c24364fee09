"""The host-buffer pipeline (slorr_pipeline_forward_backward): weights and grads
in page-locked host memory, copied in and out per group of matrices while other
groups are regularized.  The regularizer is a sum of independent per-matrix
terms (Sec. 3), so the pipeline must reproduce the device-resident call
exactly: per-matrix values and accumulated grads bit for bit, the loss up to
the order in which the groups' partial losses are added (1e-6 relative)."""

import numpy as np
import pytest

import oracle
import workloads

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

SHAPES = [(64, 147), (256, 768), (768, 256), (320, 1280), (1000, 512), (130, 700), (384, 384), (640, 1000),
          (64, 64)]


@pytest.fixture(scope="module", autouse=True)
def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2607_08754_gb300 import slorr
    slorr.load_library()


def _host(arrs):
    return [torch.from_numpy(a).pin_memory() for a in arrs]


@pytest.mark.parametrize("groups", [1, 3, 8, 100])
def test_pipeline_equals_device_call(groups):
    from paper_2607_08754_gb300.slorr import Regularizer, Pipeline
    Ws = [workloads.random_matrix(s, seed=300 + i, std=0.05) for i, s in enumerate(SHAPES)]
    G0 = [workloads.random_matrix(s, seed=400 + i, std=0.01) for i, s in enumerate(SHAPES)]
    # device-resident reference call
    reg = Regularizer(SHAPES, lam=0.3)
    w = [torch.from_numpy(W).cuda() for W in Ws]
    g = [torch.from_numpy(G).cuda() for G in G0]
    per = torch.empty(len(SHAPES), device="cuda")
    loss = reg(w, g, per_matrix=per).item()
    torch.cuda.synchronize()
    assert reg.status() == 0
    # pipelined call, twice (the grads accumulate)
    pipe = Pipeline(SHAPES, groups=groups, lam=0.3)
    hw, hg = _host(Ws), _host(G0)
    dw = [torch.empty_like(x) for x in w]
    dg = [torch.empty_like(x) for x in w]
    hl = torch.zeros(1).pin_memory()
    hp = torch.zeros(len(SHAPES)).pin_memory()
    pipe(hw, hg, dw, dg, hl, hp)
    torch.cuda.synchronize()
    assert pipe.status() == 0
    assert hl.item() == pytest.approx(loss, rel=1e-6)
    assert torch.equal(hp, per.cpu())
    for a, b in zip(hg, g):
        assert torch.equal(a, b.cpu())
    pipe(hw, hg, dw, dg, hl, hp)
    reg(w, g)
    torch.cuda.synchronize()
    for a, b in zip(hg, g):
        assert torch.equal(a, b.cpu())
    for a, W in zip(hw, Ws):   # the weights are only read
        assert torch.equal(a, torch.from_numpy(W))


def test_pipeline_vit_b16_matches_oracle_sampled():
    """The bench's e2e configuration on the ViT-B/16 set: sampled matrices
    against the fp64 oracle at the fp16-mode tolerance (2e-2)."""
    from paper_2607_08754_gb300.slorr import Pipeline
    name = "vit_b16"
    shapes = workloads.shapes(name)
    Ws = workloads.generate(name)
    pipe = Pipeline(shapes, groups=8)
    hw = _host(Ws)
    hg = [torch.zeros(s).pin_memory() for s in shapes]
    dw = [torch.empty(s, device="cuda") for s in shapes]
    dg = [torch.empty(s, device="cuda") for s in shapes]
    hl = torch.zeros(1).pin_memory()
    hp = torch.zeros(len(shapes)).pin_memory()
    pipe(hw, hg, dw, dg, hl, hp)
    torch.cuda.synchronize()
    assert pipe.status() == 0
    assert hl.item() == pytest.approx(float(hp.double().sum()), rel=1e-6)
    co = oracle.pe_coefficients(6)
    for i in (0, 5, 22, 47):
        L, G, _, _ = oracle.reg_single(Ws[i].astype(np.float64), "hoyer", co)
        assert abs(hp[i].item() - L) <= 2e-2 * L
        got = hg[i].double().numpy()
        assert np.linalg.norm(got - G) <= 2e-2 * np.linalg.norm(G), i


@pytest.mark.parametrize("dtype,variant,flags,compute", [("bf16", "hoyer", 0, "fp16"), ("f32", "nuclear", 0, "fp16"),
                                                         ("f32", "hoyer", 32, "fp16"), ("bf16", "nuclear", 32, "fp16"),
                                                         ("f32", "hoyer", 0, "bf16_split")])
def test_pipeline_options_equal_device_call(dtype, variant, flags, compute):
    """bf16 weight storage, the nuclear variant, SLORR_FLAG_WRITE_GRAD (32) and
    the bf16 hi/lo operand mode go through the pipeline unchanged: grads and
    per-matrix values equal the device-resident call bit for bit."""
    from paper_2607_08754_gb300.slorr import Regularizer, Pipeline
    tdt = torch.float32 if dtype == "f32" else torch.bfloat16
    Ws = [torch.from_numpy(workloads.random_matrix(s, seed=700 + i, std=0.05)).to(tdt) for i, s in enumerate(SHAPES)]
    G0 = [torch.from_numpy(workloads.random_matrix(s, seed=800 + i, std=0.01)).to(tdt) for i, s in enumerate(SHAPES)]
    kw = dict(variant=variant, dtype=dtype, flags=flags, lam=0.7, compute=compute)
    reg = Regularizer(SHAPES, **kw)
    w = [x.cuda() for x in Ws]
    g = [x.cuda() for x in G0]
    per = torch.empty(len(SHAPES), device="cuda")
    loss = reg(w, g, per_matrix=per).item()
    torch.cuda.synchronize()
    assert reg.status() == 0
    pipe = Pipeline(SHAPES, groups=3, **kw)
    hw = [x.pin_memory() for x in Ws]
    hg = [x.clone().pin_memory() for x in G0]
    dw = [torch.empty_like(x) for x in w]
    dg = [torch.empty_like(x) for x in w]
    hl = torch.zeros(1).pin_memory()
    hp = torch.zeros(len(SHAPES)).pin_memory()
    pipe(hw, hg, dw, dg, hl, hp)
    torch.cuda.synchronize()
    assert pipe.status() == 0
    assert hl.item() == pytest.approx(loss, rel=1e-6)
    assert torch.equal(hp, per.cpu())
    for a, b in zip(hg, g):
        assert torch.equal(a, b.cpu())
