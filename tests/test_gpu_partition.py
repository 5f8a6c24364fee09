"""App. F through the library: the regularized layers partitioned across
data-parallel ranks, each rank running libslorr on its own subset with
grad_scale = world, the existing gradient average then restoring lambda.

On one GPU the ranks are run one after another (they never wait on one
another: the only exchange is the gradient average, a host-side sum here and
a gloo all-reduce of CPU tensors in the multi-process test).  The averaged,
partitioned gradients must equal the whole-set call: bit for bit for world 2
(scaling by 2 and dividing by 2 are exact) with unsplit Gram tiles, whose
per-matrix arithmetic does not depend on which other matrices share the
launch; within fp32 rounding for world 3; and within the parity tolerance of
the oracle either way."""

import os
import socket

import numpy as np
import pytest

import oracle
import workloads

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

EPS = 1e-7


@pytest.fixture(scope="module", autouse=True)
def _need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2607_08754_gb300 import slorr
    slorr.load_library()   # raises if the extension is missing: no fallback


def call(shapes, Ws, lam, grad_scale=1.0, flags=0):
    from paper_2607_08754_gb300.slorr import Regularizer
    reg = Regularizer(shapes, lam=lam, grad_scale=grad_scale, flags=flags)
    w = [torch.from_numpy(W).cuda() for W in Ws]
    g = [torch.zeros_like(x) for x in w]
    per = torch.empty(len(Ws), device="cuda")
    loss = reg(w, g, per_matrix=per).item()
    torch.cuda.synchronize()
    assert reg.status() == 0
    return loss, per.cpu().numpy(), [x.cpu() for x in g]


def partitioned(shapes, Ws, world, lam, flags=0):
    """Every rank's call on its subset, then the data-parallel average of the
    gradients (each matrix has exactly one owner) and the sum of the losses."""
    from paper_2607_08754_gb300.slorr import slorr_partition
    grads = [torch.zeros(s, dtype=torch.float32) for s in shapes]
    per = np.full(len(shapes), np.nan, np.float32)
    loss = 0.0
    owners = []
    for r in range(world):
        mine = slorr_partition(shapes, world, r)
        owners.append(mine)
        l, p, g = call([shapes[i] for i in mine], [Ws[i] for i in mine], lam, float(world), flags)
        loss += l
        for k, i in enumerate(mine):
            grads[i] += g[k]
            per[i] = p[k]
    assert sorted(i for o in owners for i in o) == list(range(len(shapes)))
    return loss, per, [g / world for g in grads]


@pytest.mark.parametrize("world", [2, 3])
@pytest.mark.parametrize("name", ["resnet18", "vit_b16"])
def test_partition_equals_whole_set(world, name):
    from paper_2607_08754_gb300.slorr import FLAG_NO_SPLIT_K
    idx = range(21) if name == "resnet18" else range(12)
    Ws = workloads.generate(name, idx)
    shapes = [W.shape for W in Ws]
    lam = 0.25
    for flags in (FLAG_NO_SPLIT_K, 0):
        ref_loss, ref_per, ref_g = call(shapes, Ws, lam, 1.0, flags)
        loss, per, grads = partitioned(shapes, Ws, world, lam, flags)
        assert loss == pytest.approx(ref_loss, rel=1e-6)
        if flags == FLAG_NO_SPLIT_K:
            assert np.array_equal(per, ref_per)
            for a, b in zip(grads, ref_g):
                if world == 2:
                    assert torch.equal(a, b)
                else:
                    assert torch.allclose(a, b, rtol=1e-6, atol=1e-6 * b.abs().max().item())
    # and the oracle, on the default plan
    co = oracle.pe_coefficients(6)
    for i in (0, len(Ws) // 2, len(Ws) - 1):
        L, G, _, _ = oracle.reg_single(Ws[i].astype(np.float64), "hoyer", co, EPS)
        assert abs(per[i] - L) <= 2e-2 * L
        assert np.linalg.norm(grads[i].double().numpy() - lam * G) <= 2e-2 * lam * np.linalg.norm(G)


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, name, q):
    """One data-parallel rank: libslorr on its own layers (cuda:0), then the
    gradient average and the loss sum over gloo, as a DDP step would do."""
    import torch
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    from paper_2607_08754_gb300.slorr import Regularizer, slorr_partition
    Ws = workloads.generate(name, range(12))
    shapes = [W.shape for W in Ws]
    mine = slorr_partition(shapes, world, rank)
    reg = Regularizer([shapes[i] for i in mine], lam=0.25, grad_scale=float(world))
    w = [torch.from_numpy(Ws[i]).cuda() for i in mine]
    g = [torch.zeros_like(x) for x in w]
    loss = reg(w, g).cpu()
    torch.cuda.synchronize()
    assert reg.status() == 0
    grads = [torch.zeros(s, dtype=torch.float32) for s in shapes]
    for k, i in enumerate(mine):
        grads[i] += g[k].cpu()
    for t in grads:
        dist.all_reduce(t)
        t /= world
    dist.all_reduce(loss)
    if rank == 0:
        q.put((loss.item(), [t.numpy() for t in grads]))
    dist.barrier()
    dist.destroy_process_group()


def test_partition_gloo_ranks_through_library():
    """Two processes (gloo, CPU all-reduce), each running libslorr on its App. F
    subset: the averaged gradients and the summed loss match the oracle."""
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, "vit_b16", q)) for r in range(2)]
    for p in procs:
        p.start()
    loss, grads = q.get(timeout=300)
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    Ws = workloads.generate("vit_b16", range(12))
    co = oracle.pe_coefficients(6)
    ref_loss, _, ref = oracle.reg_forward_backward([W.astype(np.float64) for W in Ws], "hoyer", co, 0.25, EPS)
    assert abs(loss - ref_loss) <= 2e-2 * ref_loss
    for g, r in zip(grads, ref):
        assert np.linalg.norm(g - r) <= 2e-2 * np.linalg.norm(r)
