"""Rank-split over two processes (gloo): the host-side slicing of the packed
factors and the all-reduce reproduce the unsplit layer. In the CPU test each
process evaluates its slice with the FP64 oracle; in the GPU test each runs
the library's forward on its slice (both processes on the one GPU) and the
FP32 partials are all-reduced through host copies."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from oracle import af1_oracle as O
import synth


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _load_rank_split():
    # The module holds no compiled code; load it without the package's
    # extension so the test also runs where the library is not built.
    import importlib.util
    here = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    spec = importlib.util.spec_from_file_location("rank_split", os.path.join(here, "paper_2609_06161_gb300", "rank_split.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_rank_slices_cover_and_align():
    rs = _load_rank_split()
    for r in (1, 127, 128, 129, 800, 2028, 3167, 6352):
        for world in (1, 2, 3, 4, 8):
            sl = rs.rank_slices(r, world)
            assert len(sl) == world
            assert sl[0][0] == 0 and sl[-1][1] == r
            for (a0, a1), (b0, b1) in zip(sl, sl[1:]):
                assert a1 == b0
            for r0, r1 in sl:
                assert r0 <= r1 and (r0 == r1 or r0 % 128 == 0)


def _worker(rank, world, port, shape, seed, result):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    rs = _load_rank_split()
    m, n, r, T = shape
    d = synth.layer_words(seed, m, n, r, T)
    Uw, Vw = torch.from_numpy(d["Uw"].view(np.int32)), torch.from_numpy(d["Vw"].view(np.int32))
    s = torch.from_numpy(d["s"].view(np.int16))
    r0, r1 = rs.rank_slices(r, world)[rank]
    y = torch.zeros((T, m), dtype=torch.float64)
    if r1 > r0:
        Uw_g, Vw_g, s_g = rs.slice_packed(Uw, Vw, s, r0, r1)
        y = torch.from_numpy(O.forward_from_packed(Uw_g.numpy().view(np.uint32), Vw_g.numpy().view(np.uint32),
                                                   d["a"], s_g.numpy().view(np.uint16), d["b"], d["x"],
                                                   m, n, r1 - r0))
    dist.all_reduce(y, op=dist.ReduceOp.SUM)
    if rank == 0:
        ref = O.forward_from_packed(d["Uw"], d["Vw"], d["a"], d["s"], d["b"], d["x"], m, n, r)
        result.put(float(np.max(np.abs(y.numpy() - ref)) / max(1e-300, float(np.max(np.abs(ref))))))
    dist.destroy_process_group()


@pytest.mark.parametrize("shape,world", [((96, 160, 300, 3), 2), ((64, 200, 129, 2), 2), ((40, 72, 100, 1), 2)])
def test_rank_split_sum_matches_unsplit(shape, world):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(g, world, port, shape, 11, q)) for g in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    err = q.get(timeout=10)
    assert err < 1e-12, err


def _gpu_worker(rank, world, port, shape, seed, result):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import paper_2609_06161_gb300 as P
    from paper_2609_06161_gb300 import rank_split as rs
    torch.cuda.set_device(0)
    m, n, r, T = shape
    d = synth.layer_words(seed, m, n, r, T)
    Uw = torch.from_numpy(d["Uw"].view(np.int32)).cuda()
    Vw = torch.from_numpy(d["Vw"].view(np.int32)).cuda()
    s = torch.from_numpy(d["s"].view(np.float16)).cuda()
    a = torch.from_numpy(d["a"].view(np.float16)).cuda()
    b = torch.from_numpy(d["b"].view(np.float16)).cuda()
    x = torch.zeros((T, n + (-n) % 8), dtype=torch.float16, device="cuda")  # rows padded to 16 bytes
    x[:, :n] = torch.from_numpy(d["x"].view(np.float16)).cuda().reshape(T, n)
    r0, r1 = rs.rank_slices(r, world)[rank]
    layer = None
    if r1 > r0:
        Uw_g, Vw_g, s_g = rs.slice_packed(Uw, Vw, s, r0, r1)
        layer = P.Layer.from_words(Uw_g, Vw_g, a, s_g, b, m, n, r1 - r0, any_rank=True)
    y32 = torch.empty((T, m + (-m) % 4), dtype=torch.float32, device="cuda")
    ws = layer.make_workspace(T) if layer is not None else None
    rs.forward_rank_split(layer, x, y32, ws, host_reduce=True)
    torch.cuda.synchronize()
    if rank == 0:
        ref = O.forward_from_packed(d["Uw"], d["Vw"], d["a"], d["s"], d["b"], d["x"], m, n, r)
        result.put(O.rowwise_rel_err(y32[:, :m].double().cpu().numpy(), ref))
    if layer is not None:
        layer.free()
    dist.destroy_process_group()


@pytest.mark.gpu
@pytest.mark.parametrize("shape", [(1024, 4096, 800, 1), (4096, 4096, 2028, 4), (700, 900, 333, 17)])
def test_rank_split_through_the_library(shape):
    """Two processes each run af1_linear_forward on their 128-aligned rank
    slice (on the same GPU; no kernel waits on another); the all-reduced FP32
    partials match the unsplit layer's oracle within the bar."""
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_gpu_worker, args=(g, 2, port, shape, 13, q)) for g in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(300)
        assert p.exitcode == 0
    err = q.get(timeout=10)
    assert err <= 2e-3, err
