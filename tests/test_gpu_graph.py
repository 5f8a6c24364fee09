"""SLORR_FLAG_GRAPH: a call's launches captured once into a CUDA graph and
replayed.  The replays run the same kernels on the same workspace, so the
results equal the direct launches bit for bit, including when the weight and
gradient tensors change between calls (their pointers are read from the
workspace) and when the outputs change (a new capture)."""

import numpy as np
import pytest

import workloads

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

SHAPES = [(256, 768), (768, 256), (130, 700), (64, 147), (512, 4608)]


@pytest.fixture(scope="module", autouse=True)
def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2607_08754_gb300 import slorr
    slorr.load_library()


@pytest.mark.parametrize("compute", ["fp16", "bf16_split"])
def test_graph_replays_equal_direct_launches(compute):
    from paper_2607_08754_gb300.slorr import Regularizer, FLAG_GRAPH
    Ws = [workloads.random_matrix(s, seed=600 + i, std=0.05) for i, s in enumerate(SHAPES)]
    outs = []
    for flags in (0, FLAG_GRAPH):
        reg = Regularizer(SHAPES, compute=compute, flags=flags, lam=0.5)
        w = [torch.from_numpy(W).cuda() for W in Ws]
        g = [torch.zeros_like(x) for x in w]
        per = torch.empty(len(SHAPES), device="cuda")
        losses, pers = [], []
        for _ in range(3):                     # accumulating into the same .grad
            losses.append(reg(w, g, per_matrix=per).clone())
            pers.append(per.clone())
        g2 = [torch.ones_like(x) for x in w]   # new grad tensors: same graph
        losses.append(reg(w, g2).clone())      # no per-matrix output: a new graph
        w3 = [x * 2 for x in w]                # new weight tensors (L(2W) = L(W))
        losses.append(reg(w3, g2, per_matrix=per).clone())
        torch.cuda.synchronize()
        assert reg.status() == 0
        outs.append(([x.cpu() for x in g + g2], torch.cat(losses).cpu(), torch.stack(pers).cpu()))
    for a, b in zip(outs[0][0], outs[1][0]):
        assert torch.equal(a, b)
    assert torch.equal(outs[0][1], outs[1][1])
    assert torch.equal(outs[0][2], outs[1][2])


def test_graph_descent_steps_equal_direct_launches():
    from paper_2607_08754_gb300.slorr import Regularizer, FLAG_GRAPH
    Ws = [workloads.random_matrix(s, seed=620 + i, std=0.05) for i, s in enumerate(SHAPES)]
    outs = []
    for flags in (0, FLAG_GRAPH):
        reg = Regularizer(SHAPES, flags=flags)
        w = [torch.from_numpy(W).cuda() for W in Ws]
        losses = [reg.descent_step(w, 0.01).clone() for _ in range(4)]
        losses.append(reg.descent_step(w, 0.02).clone())   # another eta: a new graph
        torch.cuda.synchronize()
        assert reg.status() == 0
        outs.append(([x.cpu() for x in w], torch.cat(losses).cpu()))
    for a, b in zip(outs[0][0], outs[1][0]):
        assert torch.equal(a, b)
    assert torch.equal(outs[0][1], outs[1][1])
    assert np.all(np.isfinite(outs[1][1].numpy()))
