"""Multi-rank host logic on CPU: two gloo ranks (world_size 2, spawned processes).

* Point sharding (App. G.4): each rank slices its own point range without
  normalising (the oracle stands in for fs_slice_fwd on the rank's GPU). The
  unnormalised numerators and weight sums are summed across ranks with
  sharding.allreduce_partials, then finalised. The result must equal the
  unsharded oracle, and so must each rank's deslice of its own points with
  the reduced tokens.
* The sharded backward: each rank's deslice backward of its points gives a
  partial d_tokens_mixed, summed across ranks (sharding.allreduce_sums); the mix
  backward then runs on the global tokens, the slice backward on the rank's
  points, and dW, dbias, dtau are summed at the end.  Every gradient must equal
  the unsharded oracle's (dx_mid and dfx on the rank's own points).
* Job timing: the job time is the maximum of the ranks' times, and the
  job rate counts every rank's points.
"""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2609_32525_gb300 import sharding

WORLD = 2


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, port, results):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=WORLD)
    try:
        from oracle import flashslice_oracle as orc
        from paper_2609_32525_gb300.workloads import make_case

        wl = make_case(2, 1001, 3, 8, 7, dtype="f32", seed=41, backward=True)
        n0, n1 = sharding.point_range(wl.N, rank, WORLD)
        local = orc.slice_fwd(wl.x_mid[:, n0:n1], wl.fx[:, n0:n1], wl.W_slice, wl.bias, wl.tau, eps=wl.eps,
                              finalize=False)
        U = torch.from_numpy(local["tokens"].copy())
        S = torch.from_numpy(local["wsum"].copy())
        sharding.allreduce_partials(U, S)
        tokens = orc.slice_finalize(U.numpy(), S.numpy(), wl.eps)
        zp = orc.mix(wl.M, tokens)
        out_local = orc.deslice_fwd(wl.x_mid[:, n0:n1], wl.W_slice, wl.bias, wl.tau, zp)

        ref = orc.forward(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, wl.M, eps=wl.eps)
        ok_tokens = np.allclose(tokens, ref["tokens"], rtol=1e-12, atol=1e-14)
        ok_wsum = np.allclose(S.numpy(), ref["wsum"], rtol=1e-12, atol=1e-14)
        ok_out = np.allclose(out_local, ref["out"][:, n0:n1], rtol=1e-12, atol=1e-14)

        # backward: exchange the partial d_tokens_mixed, then the parameter gradients
        x_l, f_l = wl.x_mid[:, n0:n1], wl.fx[:, n0:n1]
        rd = orc.deslice_bwd(x_l, wl.W_slice, wl.bias, wl.tau, zp, wl.dout[:, n0:n1])
        dzm = torch.from_numpy(np.ascontiguousarray(rd["d_tokens_mixed"]))
        sharding.allreduce_sums(dzm)
        rm = orc.mix_bwd(wl.M, tokens, dzm.numpy())
        rs = orc.slice_bwd(x_l, f_l, wl.W_slice, wl.bias, wl.tau, tokens, S.numpy(), rm["d_tokens"], eps=wl.eps)
        grads = [torch.from_numpy(np.ascontiguousarray(rd[k] + rs[k])) for k in ("dW", "dbias", "dtau")]
        sharding.allreduce_sums(*grads)
        rb = orc.backward(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, wl.M, wl.dout, eps=wl.eps)

        def close(a, b):
            return np.allclose(a, b, rtol=1e-10, atol=1e-12)

        ok_bwd = {"dM": close(rm["dM"], rb["dM"]),
                  "dx_mid": close(rd["dx_mid"] + rs["dx_mid"], rb["dx_mid"][:, n0:n1]),
                  "dfx": close(rs["dfx"], rb["dfx"][:, n0:n1]),
                  **{k: close(g.numpy(), rb[k]) for k, g in zip(("dW", "dbias", "dtau"), grads)}}
        t = sharding.job_time_ms(1.0 + rank)
        results[rank] = (ok_tokens, ok_wsum, ok_out, t, (n0, n1), ok_bwd)
    finally:
        dist.destroy_process_group()


class _OracleOps:
    """The local compute of sharding.sharded_forward / sharded_backward on a CPU rank:
    the fp64 oracle on this rank's points, standing in for flashslice.ShardedCoupling
    (the same call sequence the C ABI runs on a GPU)."""

    def __init__(self, wl, n0, n1):
        from oracle import flashslice_oracle as orc

        self.orc, self.wl = orc, wl
        self.x, self.f, self.do = wl.x_mid[:, n0:n1], wl.fx[:, n0:n1], wl.dout[:, n0:n1]

    def slice_partials(self):
        wl = self.wl
        r = self.orc.slice_fwd(self.x, self.f, wl.W_slice, wl.bias, wl.tau, eps=wl.eps, finalize=False)
        return torch.from_numpy(r["tokens"].copy()), torch.from_numpy(r["wsum"].copy())

    def finalize(self, U, S):
        self.S = S.numpy()
        self.tokens = self.orc.slice_finalize(U.numpy(), self.S, self.wl.eps)
        return self.tokens

    def mix(self, tokens):
        self.zp = self.orc.mix(self.wl.M, tokens)
        return self.zp

    def deslice(self, zp):
        wl = self.wl
        self.out = self.orc.deslice_fwd(self.x, wl.W_slice, wl.bias, wl.tau, zp)
        return self.out

    def deslice_bwd(self):
        wl = self.wl
        self.rd = self.orc.deslice_bwd(self.x, wl.W_slice, wl.bias, wl.tau, self.zp, self.do)
        return torch.from_numpy(np.ascontiguousarray(self.rd["d_tokens_mixed"]))

    def mix_bwd(self, dzp):
        rm = self.orc.mix_bwd(self.wl.M, self.tokens, dzp.numpy())
        return rm["d_tokens"], rm["dM"]

    def slice_bwd(self, dz):
        wl = self.wl
        self.rs = self.orc.slice_bwd(self.x, self.f, wl.W_slice, wl.bias, wl.tau, self.tokens, self.S, dz, eps=wl.eps)
        return tuple(torch.from_numpy(np.ascontiguousarray(self.rd[k] + self.rs[k])) for k in ("dW", "dbias", "dtau"))


def _orchestration_worker(rank, port, results):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=WORLD)
    try:
        from oracle import flashslice_oracle as orc
        from paper_2609_32525_gb300.workloads import make_case

        wl = make_case(2, 777, 2, 8, 6, dtype="f32", seed=43, backward=True)
        n0, n1 = sharding.point_range(wl.N, rank, WORLD)
        ops = _OracleOps(wl, n0, n1)
        out = sharding.sharded_forward(ops)
        dM, (dW, db, dt) = sharding.sharded_backward(ops)
        ref = orc.forward(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, wl.M, eps=wl.eps)
        rb = orc.backward(wl.x_mid, wl.fx, wl.W_slice, wl.bias, wl.tau, wl.M, wl.dout, eps=wl.eps)

        def close(a, b):
            return bool(np.allclose(a, b, rtol=1e-10, atol=1e-12))

        results[rank] = {"out": close(out, ref["out"][:, n0:n1]), "tokens": close(ops.tokens, ref["tokens"]),
                         "dM": close(dM, rb["dM"]), "dW": close(dW.numpy(), rb["dW"]),
                         "dbias": close(db.numpy(), rb["dbias"]), "dtau": close(dt.numpy(), rb["dtau"]),
                         "dx_mid": close(ops.rd["dx_mid"] + ops.rs["dx_mid"], rb["dx_mid"][:, n0:n1]),
                         "dfx": close(ops.rs["dfx"], rb["dfx"][:, n0:n1])}
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_run_the_sharded_orchestration():
    """sharding.sharded_forward and sharded_backward, the functions bench.py --shard
    runs over NCCL, on two gloo ranks with the oracle as each rank's compute: every
    output and gradient equals the unsharded oracle's."""
    port = _free_port()
    with mp.Manager() as mgr:
        results = mgr.dict()
        mp.spawn(_orchestration_worker, args=(port, results), nprocs=WORLD, join=True)
        res = dict(results)
    assert sorted(res) == list(range(WORLD))
    for rank, oks in res.items():
        bad = [k for k, ok in oks.items() if not ok]
        assert not bad, f"rank {rank}: sharded results differ from the unsharded oracle: {bad}"


def test_point_range_partitions_the_points():
    for N in (1, 7, 1000, 1001):
        for world in (1, 2, 3, 8):
            ranges = [sharding.point_range(N, r, world) for r in range(world)]
            assert ranges[0][0] == 0 and ranges[-1][1] == N
            assert all(a[1] == b[0] for a, b in zip(ranges, ranges[1:]))
            sizes = [b - a for a, b in ranges]
            assert max(sizes) - min(sizes) <= 1
    with pytest.raises(ValueError):
        sharding.point_range(10, 2, 2)


def test_single_process_job_time_and_rate():
    assert sharding.job_time_ms(3.5) == 3.5
    assert sharding.job_rate(1_000_000, 4, 10.0) == pytest.approx(400.0)


def test_two_gloo_ranks_shard_points_forward_backward_and_time_the_job():
    port = _free_port()
    with mp.Manager() as mgr:
        results = mgr.dict()
        mp.spawn(_worker, args=(port, results), nprocs=WORLD, join=True)
        res = dict(results)
    assert sorted(res) == list(range(WORLD))
    for rank, (ok_tokens, ok_wsum, ok_out, t, rng, ok_bwd) in res.items():
        assert ok_tokens and ok_wsum, f"rank {rank}: reduced tokens differ from the unsharded oracle"
        assert ok_out, f"rank {rank}: local deslice differs"
        bad = [k for k, ok in ok_bwd.items() if not ok]
        assert not bad, f"rank {rank}: sharded gradients differ from the unsharded oracle: {bad}"
        assert t == float(WORLD)  # max over ranks of 1 + rank
    assert res[0][4][1] == res[1][4][0]
