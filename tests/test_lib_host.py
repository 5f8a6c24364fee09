"""Host-side checks of libslorr (no GPU): the library loads and exports every
symbol include/slorr.h declares, its Polar Express schedule agrees with the
oracle's independently written generator, argument validation rejects bad
requests before any CUDA call, and the App. F layer partition reproduces the
single-rank gradient under a 2-rank gloo all-reduce."""

import os
import socket

import numpy as np
import pytest

import oracle
import workloads

slorr = pytest.importorskip("paper_2607_08754_gb300.slorr")


@pytest.fixture(scope="module")
def lib():
    try:
        return slorr.load_library()
    except ImportError as e:  # pragma: no cover - the build step makes it
        pytest.fail(str(e))


def test_exports_every_declared_symbol(lib):
    names = slorr.declared_symbols()
    assert len(names) >= 16
    for n in names:
        assert hasattr(lib, n), n


@pytest.mark.parametrize("T", [1, 2, 4, 6, 8, 10])
def test_schedule_matches_oracle(lib, T):
    got = slorr.slorr_pe_coefficients(T)
    ref = oracle.pe_coefficients(T=T)
    assert np.allclose(got, ref, rtol=1e-9, atol=1e-12)


@pytest.mark.parametrize("cushion,safety", [(0.0, 1.0), (0.0, 1.01), (-1.0, 1.0), (0.05, 1.02)])
def test_schedule_options_match_oracle(lib, cushion, safety):
    got = slorr.slorr_pe_coefficients(6, 1e-3, cushion, safety)
    ref = oracle.pe_coefficients(T=6, cushion=None if cushion < 0 else cushion, safety=safety)
    assert np.allclose(got, ref, rtol=1e-10)


def test_cushion_ratio(lib):
    assert slorr.slorr_cushion_ratio() == pytest.approx(oracle.cushion_ratio(), rel=1e-12)


def test_handle_coefficients_and_flops(lib):
    shapes = workloads.shapes("vit_l16")
    r = slorr.Regularizer(shapes)
    assert np.allclose(r.coefficients(), oracle.pe_coefficients(6), rtol=1e-9)
    assert slorr.slorr_flops(shapes, 6) == oracle.weight_set_flops(shapes, 6)
    # ViT-L/16: 8659 GFLOP per step at T = 6 (paper's count, Sec. 3)
    assert slorr.slorr_flops(shapes, 6) / 1e9 == pytest.approx(8659.0, rel=1e-3)


def test_validation_rejects_bad_requests(lib):
    with pytest.raises(slorr.SlorrError) as e:
        slorr.slorr_create([(0, 3)])
    assert e.value.status == 1
    with pytest.raises(slorr.SlorrError):
        slorr.slorr_create([(3, 70000)])
    for field, bad in [("iters", 0), ("iters", 17), ("ell", 0.0), ("ell", 1.0), ("safety", 0.5),
                       ("eps", -1.0), ("variant", 5), ("compute", 9), ("dtype", 3), ("timeout_s", 0.0),
                       ("flags", 2), ("flags", 8192), ("flags", 1 << 20)]:
        o = slorr.slorr_default_options()
        setattr(o, field, bad)
        with pytest.raises(slorr.SlorrError) as e:
            slorr.slorr_create([(4, 4)], o)
        assert e.value.status == 1, field
    h = slorr.slorr_create([(4, 4)])
    ws = slorr.slorr_workspace_size(h)
    # NULL / misaligned pointers and a short workspace are rejected before any launch
    with pytest.raises(slorr.SlorrError) as e:
        slorr.slorr_reg_forward_backward(h, [0], [256], 512, 0, 1024, ws, 0)
    assert e.value.status == 1
    with pytest.raises(slorr.SlorrError) as e:
        slorr.slorr_reg_forward_backward(h, [8], [256], 512, 0, 1024, ws, 0)
    assert e.value.status == 1
    with pytest.raises(slorr.SlorrError) as e:
        slorr.slorr_reg_forward_backward(h, [256], [256], 512, 0, 1024, ws, 0)
    assert e.value.status == 1       # grad aliases weight
    with pytest.raises(slorr.SlorrError) as e:
        slorr.slorr_reg_forward_backward(h, [256], [512], 768, 0, 1024, ws - 1, 0)
    assert e.value.status == 4
    with pytest.raises(slorr.SlorrError) as e:
        slorr.slorr_reg_forward_backward(h, [256], [512], 768, 0, 1030, ws, 0)
    assert e.value.status == 4       # misaligned workspace
    # the in-place descent step: a non-finite step, a NULL loss, a short workspace
    for eta in [float("nan"), float("inf"), -float("inf")]:
        with pytest.raises(slorr.SlorrError) as e:
            slorr.slorr_reg_descent_step(h, [256], eta, 768, 0, 1024, ws, 0)
        assert e.value.status == 1 and "eta" in str(e.value)
    with pytest.raises(slorr.SlorrError) as e:
        slorr.slorr_reg_descent_step(h, [256], 0.1, 0, 0, 1024, ws, 0)
    assert e.value.status == 1
    with pytest.raises(slorr.SlorrError) as e:
        slorr.slorr_reg_descent_step(h, [256], 0.1, 768, 0, 1024, ws - 1, 0)
    assert e.value.status == 4
    slorr.slorr_destroy(h)
    o = slorr.slorr_default_options()
    o.lambda_ = 1e30
    h = slorr.slorr_create([(4, 4)], o)
    with pytest.raises(slorr.SlorrError) as e:
        slorr.slorr_reg_descent_step(h, [256], 1e30, 768, 0, 1024, slorr.slorr_workspace_size(h), 0)
    assert e.value.status == 1 and "overflows" in str(e.value)
    slorr.slorr_destroy(h)


def test_workspace_size_grows_with_the_set(lib):
    small = slorr.Regularizer([(64, 64)]).workspace_bytes
    big = slorr.Regularizer([(64, 64), (1000, 512)]).workspace_bytes
    fp32 = slorr.Regularizer([(64, 64), (1000, 512)], compute="fp32").workspace_bytes
    assert small < big < fp32
    # X0, X1 (Ppad x Qpad) and A, B (Ppad x Ppad) of 1000x512 in fp16 alone:
    assert big - small >= 2 * (512 * 1024 * 2) + 2 * (512 * 512 * 2)


def test_partition_is_a_balanced_cover(lib):
    shapes = workloads.shapes("decoder_560m")
    for world in (1, 2, 3, 8):
        parts = [slorr.slorr_partition(shapes, world, r) for r in range(world)]
        flat = sorted(i for p in parts for i in p)
        assert flat == list(range(len(shapes)))
        loads = [sum(oracle.pe_flops(*shapes[i]) for i in p) for p in parts]
        assert max(loads) <= min(loads) + max(oracle.pe_flops(*s) for s in shapes)


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _partition_worker(rank, world, port, shapes, q):
    import torch
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    from paper_2607_08754_gb300 import slorr as sl
    mine = sl.slorr_partition(shapes, world, rank)
    co = oracle.pe_coefficients(6)
    Ws = [np.random.default_rng(50 + i).normal(size=s) for i, s in enumerate(shapes)]
    grads = [torch.zeros(s, dtype=torch.float64) for s in shapes]
    loss = torch.zeros(1, dtype=torch.float64)
    sub = [Ws[i] for i in mine]
    l, _, incs = oracle.reg_forward_backward(sub, "hoyer", co, lam=0.3, grad_scale=float(world))
    for i, g in zip(mine, incs):
        grads[i] += torch.from_numpy(g)
    loss += l
    for g in grads:                      # the data-parallel gradient average
        dist.all_reduce(g)
        g /= world
    dist.all_reduce(loss)                # logged loss: plain sum
    if rank == 0:
        q.put((loss.item(), [g.numpy() for g in grads]))
    dist.barrier()
    dist.destroy_process_group()


def test_layer_partition_two_ranks_gloo(lib):
    """App. F: each rank regularizes its layers with grad_scale = world; the
    data-parallel average then equals the single-rank gradient."""
    import torch.multiprocessing as mp
    shapes = [(6, 9), (12, 5), (7, 7), (3, 11), (10, 4)]
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_partition_worker, args=(r, 2, port, shapes, q)) for r in range(2)]
    for p in procs:
        p.start()
    loss, grads = q.get(timeout=120)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    co = oracle.pe_coefficients(6)
    Ws = [np.random.default_rng(50 + i).normal(size=s) for i, s in enumerate(shapes)]
    ref_loss, _, ref = oracle.reg_forward_backward(Ws, "hoyer", co, lam=0.3)
    assert loss == pytest.approx(ref_loss, rel=1e-12)
    for g, r in zip(grads, ref):
        assert np.allclose(g, r, rtol=1e-12, atol=1e-15)


def test_pipeline_validation_and_workspace(lib):
    """The host-buffer pipeline rejects bad requests before any CUDA call, and
    its workspace holds every group's plan."""
    shapes = [(64, 576), (128, 1152), (256, 2304), (512, 4608), (1000, 512)]
    with pytest.raises(slorr.SlorrError) as e:
        slorr.slorr_pipeline_create(shapes, None, 0)
    assert e.value.status == 1
    with pytest.raises(slorr.SlorrError):
        slorr.slorr_pipeline_create([(0, 4)], None, 2)
    single = slorr.slorr_workspace_size(slorr.slorr_create(shapes))
    for groups in (1, 2, 5, 50):
        p = slorr.slorr_pipeline_create(shapes, None, groups)
        ws = slorr.slorr_pipeline_workspace_size(p)
        assert ws >= single - 1024 * groups   # each group carries its own plan
        with pytest.raises(slorr.SlorrError) as e:   # NULL host pointer
            slorr.slorr_pipeline_forward_backward(p, [256] * 4 + [0], [512] * 5, 768, 0, [1024] * 5, [2048] * 5,
                                                  4096, ws, 0)
        assert e.value.status == 1
        with pytest.raises(slorr.SlorrError) as e:   # short workspace
            slorr.slorr_pipeline_forward_backward(p, [256] * 5, [512] * 5, 768, 0, [1024] * 5, [2048] * 5,
                                                  4096, ws - 1, 0)
        assert e.value.status == 4
        slorr.slorr_pipeline_destroy(p)


def test_executed_flops_counts_pair_tiles(lib):
    """slorr_executed_flops: 2 x 256 x nsz x K over the CTA-pair tiles of every
    phase (P and Q padded to multiples of 128, strictly-lower 256 x 256 tiles of
    the symmetric Gram and Poly products skipped), times T.  A square 256 x 256
    matrix executes exactly the paper's count."""
    def expected(shapes, T):
        tot = 0
        for m, n in shapes:
            P, Q = min(m, n), max(m, n)
            Pp, Qp = -(-P // 128) * 128, -(-Q // 128) * 128
            for ph, (N, K) in enumerate([(Pp, Qp), (Pp, Pp), (Qp, Pp)]):
                for tm in range(-(-Pp // 256)):
                    for tn in range(-(-N // 256)):
                        nsz = min(256, N - tn * 256)
                        if ph < 2 and tn < tm:
                            continue
                        tot += 2 * 256 * nsz * K
        return tot * T
    for shapes in ([(256, 256)], [(1000, 512)], [(64, 147), (3072, 1024), (1024, 4096), (130, 700)]):
        r = slorr.Regularizer(shapes, iters=4)
        assert slorr.slorr_executed_flops(r.handle) == expected(shapes, 4)
    assert slorr.slorr_executed_flops(slorr.Regularizer([(256, 256)]).handle) == \
        slorr.slorr_flops([(256, 256)], 6)


def test_split_k_plan(lib):
    """The Gram tiles of a set with few long-K tiles are split into K parts
    (at most 2, about max(1024, the launch's K per pair) each); sets
    whose Gram tiles already fill the pairs, Poly and Update, the
    CUDA-core path and SLORR_FLAG_NO_SPLIT_K are not.  Splitting changes
    neither the tiles' total K nor the executed FLOPs."""
    import workloads
    rn = workloads.shapes("resnet18")
    split = slorr.Regularizer(rn)
    whole = slorr.Regularizer(rn, flags=slorr.FLAG_NO_SPLIT_K)
    g_split = slorr.slorr_gemm_items(split.handle, 0)
    g_whole = slorr.slorr_gemm_items(whole.handle, 0)
    assert g_whole < g_split <= 2 * g_whole
    for ph in (1, 2):
        assert slorr.slorr_gemm_items(split.handle, ph) == slorr.slorr_gemm_items(whole.handle, ph)
    assert slorr.slorr_executed_flops(split.handle) == slorr.slorr_executed_flops(whole.handle)
    assert split.workspace_bytes > whole.workspace_bytes      # the parts' fp32 partial slots
    # one 512 x 4608 matrix alone: its 3 Gram tiles (K = 4608, 72 K blocks) become 3 x 2 parts
    one = slorr.Regularizer([(512, 4608)])
    assert slorr.slorr_gemm_items(one.handle, 0) == 6
    # the ViT-L/16 set's 960 Gram tiles fill the 76 pairs many times over
    vl = workloads.shapes("vit_l16")
    assert slorr.slorr_gemm_items(slorr.Regularizer(vl).handle, 0) == \
        slorr.slorr_gemm_items(slorr.Regularizer(vl, flags=slorr.FLAG_NO_SPLIT_K).handle, 0) == 960
    assert slorr.slorr_gemm_items(slorr.Regularizer(rn, compute="fp32").handle, 0) == \
        slorr.slorr_gemm_items(slorr.Regularizer(rn, compute="fp32", flags=slorr.FLAG_NO_SPLIT_K).handle, 0)
    with pytest.raises(slorr.SlorrError):
        slorr.slorr_gemm_items(split.handle, 3)


def expected_tiles(shapes, phase):
    """The tensor-core tiles of one phase, written out from the shapes: 256 x 256
    tiles of the padded products (P and Q padded to multiples of 128), the
    strictly-lower tiles of the symmetric Gram and Poly products left out;
    (mat, tm, tn, msz, nsz) and the tile's K."""
    out = []
    for i, (m, n) in enumerate(shapes):
        P, Q = min(m, n), max(m, n)
        Pp, Qp = -(-P // 128) * 128, -(-Q // 128) * 128
        N = Qp if phase == 2 else Pp
        K = Qp if phase == 0 else Pp
        for tm in range(-(-Pp // 256)):
            for tn in range(-(-N // 256)):
                msz, nsz = min(256, Pp - 256 * tm), min(256, N - 256 * tn)
                if phase < 2 and 2 * tn + nsz // 128 - 1 < 2 * tm:
                    continue
                out.append(((i, tm, tn, msz, nsz), K))
    return out


def pair_loads(ks, npairs=76):
    """Per-pair total K when item j goes to pair j mod npairs."""
    load = [0] * npairs
    for j, k in enumerate(ks):
        load[j % npairs] += k
    return load


def test_pair_plan_is_balanced(lib):
    """The CTA-pair kernel hands item i to pair i mod npairs; the plan orders
    its items so that the 76 pairs of a GB300 get nearly equal total K.
    ViT-L/16's Gram has 960 tiles (10 per 1024-row matrix) with K = 4096, 3072
    and 1024: sorted round-robin gives one pair 40960, the balanced order at
    most one K = 1024 tile above the ideal total / 76.  The plan's items are
    exactly the tiles written out from the shapes (as a multiset), the totals
    match, and equal-K phases reach the whole-tile optimum ceil(tiles / 76) * K."""
    import math
    import workloads
    vl = workloads.shapes("vit_l16")
    pair = slorr.Regularizer(vl)
    items = slorr.slorr_gemm_item_list(pair.handle, 0)
    exp = expected_tiles(vl, 0)
    assert sorted(map(tuple, items[:, :5].tolist())) == sorted(t for t, _ in exp)
    assert np.all(items[:, 5] == 0) and np.all(items[:, 6] == 1)   # ViT-L/16's Gram tiles are not split
    mx, tot = slorr.slorr_gemm_pair_load(pair.handle, 0)
    assert tot == sum(10 * max(s) for s in vl) == sum(k for _, k in exp)
    assert mx <= math.ceil(tot / 76) + 1024
    kmap = {t: k for t, k in exp}
    assert mx == max(pair_loads([kmap[tuple(r)] for r in items[:, :5].tolist()]))
    # the sorted order without balancing (longest K first, stable)
    srt = sorted(exp, key=lambda e: -e[1])
    assert max(pair_loads([k for _, k in srt])) == 40960 and mx < 40960
    for ph, tiles in ((1, 960), (2, 4608)):
        m, t = slorr.slorr_gemm_pair_load(pair.handle, ph)
        assert t == tiles * 1024 and m == math.ceil(tiles / 76) * 1024
    with pytest.raises(slorr.SlorrError):
        slorr.slorr_gemm_pair_load(pair.handle, 0, 0)


def test_pair_plan_balance_on_random_sets(lib):
    """On random weight sets (1 to 40 matrices, sides 1 to 3000) the CTA-pair
    plan's Gram and Update items are exactly the tiles written out from the
    shapes (compared as multisets: a dropped tile and a duplicated one with
    the same K would be caught), and its largest per-pair total over 76 pairs
    is not above that of the sorted order.  The planner weighs each tile as
    its K plus one K block (64) for its fixed cost, so in pure K the bound
    holds to within that one block."""
    rng = np.random.default_rng(2607)
    for _ in range(25):
        count = int(rng.integers(1, 41))
        shapes = [(int(rng.integers(1, 3001)), int(rng.integers(1, 3001))) for _ in range(count)]
        pair = slorr.Regularizer(shapes, flags=slorr.FLAG_NO_SPLIT_K)
        for ph in (0, 2):
            items = slorr.slorr_gemm_item_list(pair.handle, ph)
            exp = expected_tiles(shapes, ph)
            assert sorted(map(tuple, items[:, :5].tolist())) == sorted(t for t, _ in exp)
            srt = sorted(exp, key=lambda e: -e[1])
            mx = slorr.slorr_gemm_pair_load(pair.handle, ph)[0]
            assert mx <= max(pair_loads([k for _, k in srt])) + 64


def test_split_plan_items(lib):
    """Split Gram tiles (ResNet-18): every tile of the set appears once per
    part, with part indices 0 .. parts - 1 and the same number of parts on
    each of them; unsplit tiles appear once as part 0 of 1."""
    import workloads
    rn = workloads.shapes("resnet18")
    items = slorr.slorr_gemm_item_list(slorr.Regularizer(rn).handle, 0)
    exp = expected_tiles(rn, 0)
    seen = {}
    for r in items.tolist():
        seen.setdefault(tuple(r[:5]), []).append((r[5], r[6]))
    assert sorted(seen) == sorted(t for t, _ in exp)
    assert any(len(v) > 1 for v in seen.values())
    for v in seen.values():
        parts = v[0][1]
        assert len(v) == parts and sorted(p for p, _ in v) == list(range(parts))
        assert all(q == parts for _, q in v)
    with pytest.raises(slorr.SlorrError):
        slorr._check(slorr.load_library().slorr_gemm_item_list(slorr.Regularizer(rn).handle, 0, None, 0))


def test_symmetric_reads_find_stored_tiles(lib):
    """A and M are stored only in the 256 x 256 tiles the Gram and the Poly
    compute.  The readers' rule (written out again here): an operand made of
    rows of A or M in tile row t reads its 128-wide K block kb K-major from
    tile (t, kb // 2) when kb // 2 >= t, else MN-major from tile (kb // 2, t).
    Every such tile must be in the plan's item list of the phase that writes
    it, for every padded size (ragged ones included)."""
    for P in (64, 128, 200, 256, 320, 384, 640, 1000, 1024, 1536, 2048):
        shapes = [(P, P + 64), (2 * P + 7, P)]
        reg = slorr.Regularizer(shapes)
        stored = {ph: {(r[0], r[1], r[2]) for r in slorr.slorr_gemm_item_list(reg.handle, ph).tolist()}
                  for ph in (0, 1)}
        Ppad = -(-P // 128) * 128
        rows = -(-Ppad // 256)   # 256-row tiles
        nkb = Ppad // 128
        for mat in range(len(shapes)):
            def tile_of(t, kb):
                return (mat, t, kb // 2) if kb // 2 >= t else (mat, kb // 2, t)
            for t in range(rows):
                for kb in range(nkb):
                    # the Update's A operand (rows of M) and both Poly operands (rows of A)
                    assert tile_of(t, kb) in stored[1], (P, mat, t, kb)
                    assert tile_of(t, kb) in stored[0], (P, mat, t, kb)


# the planner's dependency latency, in K blocks (written out again here)
DEP = 8.0


def _df_cost(shapes, phase, nsz, K):
    """The planner's cost of one item in K blocks (written out again here)."""
    kb = (K // 64) * (0.5 + 0.5 * nsz / 256.0)
    return (1.6 * kb if phase == 1 else kb) + 1.0


@pytest.mark.parametrize("name", ["cfg1", "resnet18", "vit_b16", "vit_l16"])
def test_dataflow_plan(lib, name):
    """The dataflow plan (every Gram, Poly and Update tile of the T steps in
    one launch): each step's items are exactly the per-phase tiles; each pair's
    items are in planned start order; every item of a matrix's (step, phase)
    group starts after every item of the group before it (so the launch cannot
    deadlock); each item waits for 16 completions per item of its matrix's
    earlier groups; and the planned duration is within 15% of the larger of
    the two lower bounds, total work / 76 pairs and the longest chain of one
    matrix's phases."""
    import workloads
    shapes = workloads.shapes(name)
    T = 6
    reg = slorr.Regularizer(shapes, iters=T, flags=slorr.FLAG_DATAFLOW)
    items, npairs, makespan = slorr.slorr_dataflow_items(reg.handle)
    assert npairs == 76
    pair, seq, step, phase, mat = (items[:, k] for k in range(5))
    # the per-phase tiles, T times
    for ph in range(3):
        ref = sorted(map(tuple, slorr.slorr_gemm_item_list(reg.handle, ph)[:, [0, 1, 2, 5, 6]].tolist()))
        for t in range(T):
            sel = items[(step == t) & (phase == ph)]
            assert sorted(map(tuple, sel[:, [4, 5, 6, 7, 8]].tolist())) == ref
    assert sorted(seq.tolist()) == list(range(len(items)))
    for q in range(npairs):
        s = seq[pair == q]
        assert np.all(np.diff(s) > 0)
    counts = {}
    for ph in range(3):
        for r in slorr.slorr_gemm_item_list(reg.handle, ph).tolist():
            counts[(r[0], ph)] = counts.get((r[0], ph), 0) + 1
    for m in range(len(shapes)):
        g = (step * 3 + phase)[mat == m]
        s = seq[mat == m]
        w = items[mat == m][:, 9]
        done = 0
        for k in range(3 * T):
            assert np.all(w[g == k] == done)
            if k + 1 < 3 * T:
                assert s[g == k].max() < s[g == k + 1].min()
            done += 16 * counts[(m, k % 3)]
    # planned duration against the lower bounds (the same cost model)
    cost = {}
    total = 0.0
    for ph in range(3):
        for r in slorr.slorr_gemm_item_list(reg.handle, ph).tolist():
            P, Q = min(shapes[r[0]]), max(shapes[r[0]])
            Pp, Qp = -(-P // 128) * 128, -(-Q // 128) * 128
            K = (Qp if ph == 0 else Pp) // r[6]
            c = _df_cost(shapes, ph, r[4], K) + (2.0 if r[6] > 1 else 0.0)
            total += T * c
            cost[(r[0], ph)] = max(cost.get((r[0], ph), 0.0), c)
    chain = max(T * sum(cost[(m, ph)] + DEP for ph in range(3)) - DEP for m in range(len(shapes)))
    bound = max(total / 76, chain)
    assert bound <= makespan <= 1.15 * bound, (makespan, total / 76, chain)


def test_dataflow_plan_is_absent_for_phase_launches(lib):
    for kw in ({"flags": slorr.FLAG_PHASE_LAUNCHES}, {"compute": "fp32"}, {"flags": slorr.FLAG_SIMT_GEMM}):
        r = slorr.Regularizer([(256, 512)], **kw)
        with pytest.raises(slorr.SlorrError):
            slorr.slorr_dataflow_items(r.handle)
    with pytest.raises(slorr.SlorrError):
        slorr.Regularizer([(256, 512)], flags=slorr.FLAG_PHASE_LAUNCHES | slorr.FLAG_DATAFLOW)


def test_launch_mode_is_chosen_by_set_shape(lib):
    """Without a flag the plan takes the dataflow launch for work-bound sets
    whose per-phase launches would be short (fewer than 7 Gram tiles per
    pair), the measured winners, and per-phase launches for chain-bound sets
    (cfg1, ResNet-18) and for sets with many tiles per pair (ViT-L/16, 560M,
    ViT-H, ViT-B with 24 blocks); SLORR_FLAG_DATAFLOW forces the dataflow
    launch."""
    import workloads
    for name, m, df in (("cfg1", 0, False), ("resnet18", 0, False), ("vit_ladder_vit_ti", 0, False),
                        ("vit_ladder_vit_s", 0, True), ("vit_ladder_vit_512", 0, True), ("vit_b16", 0, True),
                        ("vit_l16", 32, True), ("vit_l16", 48, True), ("decoder_560m", 28, True),
                        ("vit_ladder_vit_b24", 0, False), ("vit_l16", 64, False), ("decoder_560m", 56, False),
                        ("vit_l16", 0, False), ("decoder_560m", 0, False), ("vit_ladder_vit_h", 0, False)):
        shapes = workloads.shapes(name)
        if m:
            shapes = shapes[:m]
        r = slorr.Regularizer(shapes)
        forced = slorr.Regularizer(shapes, flags=slorr.FLAG_DATAFLOW)
        mk = slorr.slorr_dataflow_items(forced.handle)[2]
        if df:
            assert slorr.slorr_dataflow_items(r.handle)[2] == mk
        else:
            with pytest.raises(slorr.SlorrError):
                slorr.slorr_dataflow_items(r.handle)
        # the workspace holds the dataflow plan only when it is used
        assert (forced.workspace_bytes > r.workspace_bytes) == (not df)


def test_bf16_split_mode_plan(lib):
    """SLORR_COMPUTE_BF16_SPLIT (bf16 hi/lo operands): the same tiles as
    bf16, per-phase launches only, a workspace with the low parts of X0, X1,
    A and M besides bf16's buffers, executed work of three products per
    product, and the flags it cannot serve rejected."""
    import workloads
    shapes = [(64, 147), (3072, 1024), (1024, 4096), (130, 700)]
    bf = slorr.Regularizer(shapes, compute="bf16", flags=slorr.FLAG_PHASE_LAUNCHES)
    sp = slorr.Regularizer(shapes, compute="bf16_split")
    for ph in range(3):
        assert np.array_equal(slorr.slorr_gemm_item_list(sp.handle, ph), slorr.slorr_gemm_item_list(bf.handle, ph))
    lo = 0
    for m, n in shapes:
        P, Q = min(m, n), max(m, n)
        Pp, Qp = -(-P // 128) * 128, -(-Q // 128) * 128
        lo += 2 * (2 * Pp * Qp) + 2 * (2 * Pp * Pp)
    assert sp.workspace_bytes - bf.workspace_bytes >= lo
    assert slorr.slorr_executed_flops(sp.handle) == 3 * slorr.slorr_executed_flops(bf.handle)
    # the dataflow launch is never planned, even for a set that takes it in bf16
    vb = workloads.shapes("vit_b16")
    slorr.slorr_dataflow_items(slorr.Regularizer(vb, compute="bf16").handle)
    with pytest.raises(slorr.SlorrError):
        slorr.slorr_dataflow_items(slorr.Regularizer(vb, compute="bf16_split").handle)
    for flag in (slorr.FLAG_SIMT_GEMM, slorr.FLAG_SEPARATE_NORM, slorr.FLAG_DATAFLOW):
        with pytest.raises(slorr.SlorrError) as e:
            slorr.Regularizer([(256, 512)], compute="bf16_split", flags=flag)
        assert e.value.status == 1


def test_pipeline_groups_by_operand_mode(lib):
    """The host-buffer pipeline's default grouping: about 64 MiB of weights
    per group (128 MiB with bf16 hi/lo operands, whose kernels take longer
    than the copies), between 1 and 16 groups."""
    import workloads
    vl = workloads.shapes("vit_l16")          # 1.21 GB of fp32 weights
    assert slorr.Pipeline.auto_groups(vl) == 16
    assert slorr.Pipeline.auto_groups(vl, "f32", "bf16_split") == 9
    assert slorr.Pipeline.auto_groups(vl, "bf16", "bf16_split") == 4
    assert slorr.Pipeline.auto_groups([(64, 64)]) == 1
    assert slorr.Pipeline.auto_groups(workloads.shapes("vit_b16"), "f32", "fp16") == 5
