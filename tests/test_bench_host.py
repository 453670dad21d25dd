"""Host logic of bench.py's multi-process path, on CPU: world-size-2 gloo ranks.

bench.py runs one independent replica per GPU (weak scaling).  Its only collectives are the
barrier around the timed region and the max of the step time over ranks; the reference arm
runs on rank 0 alone.  These tests exercise exactly that logic with the gloo backend."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port), "RANK": str(rank),
                       "WORLD_SIZE": str(world), "LOCAL_RANK": str(rank)})
    import bench
    import torch.distributed as dist
    r, w, local = bench.dist_setup()
    assert (r, w, local) == (rank, world, rank)
    assert dist.get_backend() == "gloo"
    bench.barrier(w)
    m = bench.max_over_ranks(0.25 + rank, w)          # per-rank step time in ms
    bench.barrier(w)
    q.put((rank, m))
    dist.destroy_process_group()


def test_two_rank_barrier_and_max_over_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
    assert all(p.exitcode == 0 for p in procs), [p.exitcode for p in procs]
    got = dict(q.get(timeout=5) for _ in range(2))
    assert got == {0: 1.25, 1: 1.25}


def test_single_process_helpers_need_no_process_group(monkeypatch):
    import bench
    for v in ("WORLD_SIZE", "RANK", "LOCAL_RANK"):
        monkeypatch.delenv(v, raising=False)
    assert bench.dist_setup() == (0, 1, 0)
    assert bench.max_over_ranks(3.5, 1) == 3.5
    bench.barrier(1)


def test_reference_arm_under_torchrun_prints_once_from_rank0():
    """--impl reference under the driver's torchrun launch: rank 0 times the oracle and prints one
    JSON line; rank 1 exits 0 without work."""
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), os.path.join(ROOT, "bench.py"),
           "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "0", "--config", "c1_256x256_k32_f32"]
    env = dict(os.environ, OMP_NUM_THREADS="2")
    out = subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [ln for ln in out.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, out.stdout
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["value"] == d["value"]
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["d2h_bytes_per_step"] == 0


def test_diagnostics_from_sums_matches_the_oracle():
    """The bench's concentration / alignment / Theorem-1 arithmetic on row-statistics sums (the
    quantities cat_block_row_stats returns) equals the oracle's analysis functions."""
    import numpy as np

    import bench
    import oracle as O
    rng = np.random.default_rng(3)
    X = rng.standard_normal((40, 24)) * rng.lognormal(0, 1, 24)
    W = rng.standard_normal((30, 24)) * 0.1
    x3 = [float(np.sum(X * X)), float(np.sum((2 * np.abs(X).max(axis=1)) ** 2))]
    w3 = [float(np.sum(W * W)), float(np.sum((2 * np.abs(W).max(axis=1)) ** 2))]
    y = X @ W.T
    dg = bench.diagnostics_from_sums(x3, w3, float(np.sum(y * y)))
    assert abs(dg["C_x_db"] - O.db(O.concentration_act(X))) < 1e-9
    assert abs(dg["C_w_db"] - O.db(O.concentration_weight(W))) < 1e-9
    assert abs(dg["A_db"] - O.db(O.alignment(X, W))) < 1e-9
    assert abs(dg["theorem1_db"] - O.db(O.theorem1_sqnr(X, W))) < 1e-9


# ------------------------------------------------------------------------------------------
# Token-sharded layer: per-rank compute by the oracle, reductions over two gloo ranks
# ------------------------------------------------------------------------------------------

class _OracleOps:
    """The per-rank computations of bench.sharded_layer_step, done by the oracle on the host."""

    def __init__(self):
        import oracle as O
        self.O = O

    def calib_cov(self, xc, k):
        return self.O.calib_cov_block_sums(xc, k)

    def quantize_weights(self, W, k, sigma_sums, n_calib):
        pw = self.O.prepare_weights(W, "cat", k, Sigma_x_blocks=sigma_sums / n_calib)
        return pw.T, pw.qw, pw.sw

    def transform_quantize_act(self, x, T, k):
        ac = self.O.transform_quantize_act(x, T)
        return ac.qx, ac.sx

    def linear_sqnr(self, qx, sx, qw, sw, y_ref):
        import numpy as np
        _, y_hat = self.O.w4a4_linear(qx, sx, qw, sw)
        sig, err = self.O.sqnr_sums(y_ref, y_hat)
        return y_hat, np.array([sig, err])


def _sharded_rank_main(rank, world, port, q):
    os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port), "RANK": str(rank),
                       "WORLD_SIZE": str(world), "LOCAL_RANK": str(rank)})
    import numpy as np
    import torch
    import torch.distributed as dist

    import bench
    import oracle as O
    import workloads as WL
    bench.dist_setup()
    cfg = WL.small_config("shard", d_in=256, d_out=160, n_eval=211, n_calib=300, k=32, seed=61)
    L = WL.make_layer(cfg)

    def allreduce_sum(arr):
        t = torch.from_numpy(np.ascontiguousarray(arr))
        dist.all_reduce(t)
        arr[...] = t.numpy()

    t0, t1 = bench.shard_range(cfg.n_eval, rank, world)
    c0, c1 = bench.shard_range(cfg.n_calib, rank, world)
    x = L.x_eval.values[t0:t1].astype(np.float64)
    y_ref = O.linear(x, L.W.values)
    y_hat, sig, err, db = bench.sharded_layer_step(_OracleOps(), x, L.x_calib.values[c0:c1].astype(np.float64), y_ref,
                                                   L.W.values, cfg.k, cfg.n_calib, allreduce_sum)
    q.put((rank, t0, t1, y_hat, sig, err, db))
    dist.destroy_process_group()


def test_token_sharded_layer_matches_one_process():
    """Two ranks each take half of the tokens (and of the calibration tokens); with the calibration
    sums and the SQNR sums all-reduced, the combined SQNR and every rank's output equal the one-process
    layer's (Sec. 6: per-token activations, per-channel weights; the layer shards by tokens)."""
    import numpy as np

    import oracle as O
    import workloads as WL
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_sharded_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = [q.get(timeout=240) for _ in range(2)]
    for p in procs:
        p.join(120)
    assert all(p.exitcode == 0 for p in procs), [p.exitcode for p in procs]
    cfg = WL.small_config("shard", d_in=256, d_out=160, n_eval=211, n_calib=300, k=32, seed=61)
    L = WL.make_layer(cfg)
    ref = O.cat_layer(L.x_eval.values, L.W.values, "cat", cfg.k, X_calib=L.x_calib.values)
    dbs = {r[6] for r in got}
    assert len(dbs) == 1                                    # every rank reports the same combined value
    assert abs(dbs.pop() - ref["sqnr_db"]) < 0.01
    for rank, t0, t1, y_hat, sig, err, db in got:
        assert abs(sig / ref["sig"] - 1) < 1e-12 and abs(err / ref["err"] - 1) < 1e-9
        np.testing.assert_allclose(y_hat, ref["y_hat"][t0:t1], rtol=1e-9, atol=1e-12)
