"""Host-side data-parallel logic on CPU: the batch split, the SUM all-reduce
of the batch-reduced gradients over gloo ranks (world size 2), and the
order of operations of a data-parallel training step.  The compute on each
rank is the oracle's, so these tests need no GPU; the GPU path differs only
in running the same steps through the library on each rank's device."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from oracle import snn_oracle as O
from paper_2211_10725_gb300 import workloads as W
from paper_2211_10725_gb300.data_parallel import (DataParallelDenseSNN, allreduce_sum_,
                                                  shard_range)


@pytest.mark.parametrize("B", [0, 1, 7, 128, 129])
@pytest.mark.parametrize("world", [1, 2, 3, 8])
def test_shard_range_partitions_the_batch(B, world):
    spans = [shard_range(B, world, r) for r in range(world)]
    assert spans[0][0] == 0 and spans[-1][1] == B
    for (a0, a1), (b0, b1) in zip(spans, spans[1:]):
        assert a1 == b0
    sizes = [b - a for a, b in spans]
    assert max(sizes) - min(sizes) <= 1 and min(sizes) >= 0


def test_shard_range_rejects_bad_arguments():
    for args in [(4, 0, 0), (4, 2, 2), (4, 2, -1), (-1, 2, 0)]:
        with pytest.raises(ValueError):
            shard_range(*args)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _dsnn_problem():
    w = W.DSNN_C3.scaled(T=4, B=6, sizes=(24, 16, 8, 5), n_classes=5)
    inp = W.make_dense_inputs(w, seed=W.SEED_BASE + 77)
    Ws = [x.float().numpy().astype(np.float64) * 3.0 for x in inp["W"]]   # enough spikes
    X = inp["X"].float().numpy().astype(np.float64)                         # [T, B, K]
    y = inp["labels"].numpy().astype(np.int64)
    return w, Ws, X, y


def _dsnn_grads(w, Ws, X, y, b0, b1, batch_total):
    """Oracle dW and loss of samples [b0, b1) with the loss averaged over
    batch_total samples (the loss kernel's normalisation)."""
    nb = b1 - b0
    xb = X[:, b0:b1].reshape(w.T * nb, -1)
    fwd = O.dsnn_forward(xb, Ws, w.T, nb, w.beta, w.thr, dtype=np.float64)
    res = O.dsnn_backward(fwd, Ws, y[b0:b1], w.T, nb, w.beta, w.thr, 5.0)
    k = nb / batch_total     # rate_ce_loss averages over nb
    return [d * k for d in res["dW"]], res["loss"] * k


def _scan_grads(w, inp, b0, b1):
    """Oracle per-neuron dbeta/dthr of lanes of samples [b0, b1)."""
    N = w.N
    I = inp["I"].float().numpy().astype(np.float64).reshape(w.T, w.B, N)[:, b0:b1].reshape(w.T, -1)
    gs = inp["grad_spk"].float().numpy().astype(np.float64).reshape(w.T, w.B, N)[:, b0:b1]
    gs = gs.reshape(w.T, -1)
    nb = b1 - b0
    beta = O.lane_param(inp["beta"].numpy(), nb, N, w.beta_mode)
    thr = O.lane_param(inp["thr"].numpy(), nb, N, w.thr_mode)
    spk, mem = O.leaky_forward(I, beta, thr, w.reset)
    g = O.leaky_backward(mem, spk, gs, beta, thr, w.reset, w.detach_reset, w.surrogate,
                         w.sg_param)
    return (O.reduce_lane_grad(g["grad_beta_lane"], nb, N, w.beta_mode),
            O.reduce_lane_grad(g["grad_thr_lane"], nb, N, w.thr_mode))


def _rank_main(rank, world, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        w, Ws, X, y = _dsnn_problem()
        b0, b1 = shard_range(w.B, world, rank)
        dW, loss = _dsnn_grads(w, Ws, X, y, b0, b1, w.B)
        flat = torch.tensor(np.concatenate([d.ravel() for d in dW] + [[loss]]))
        allreduce_sum_([flat])
        sw = W.BIG_C5.scaled(T=6, B=5, N=16)
        inp = W.make_scan_inputs(sw)
        s0, s1 = shard_range(sw.B, world, rank)
        gb, gt = _scan_grads(sw, inp, s0, s1)
        pg = [torch.tensor(gb), torch.tensor(gt)]
        allreduce_sum_(pg)
        np.savez(os.path.join(out_dir, f"rank{rank}.npz"), dsnn=flat.numpy(), gbeta=pg[0].numpy(),
                 gthr=pg[1].numpy())
    finally:
        dist.destroy_process_group()


def test_sharded_gradients_sum_to_the_full_batch(tmp_path):
    """Two gloo ranks, each on its half of the batch: after the SUM
    all-reduce every rank holds the full-batch dW, loss and per-neuron
    beta / threshold gradients of the oracle."""
    world = 2
    mp.spawn(_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True)
    w, Ws, X, y = _dsnn_problem()
    dW, loss = _dsnn_grads(w, Ws, X, y, 0, w.B, w.B)
    full = np.concatenate([d.ravel() for d in dW] + [[loss]])
    assert np.abs(full[:-1]).max() > 1e-6          # the gradients are not all zero
    sw = W.BIG_C5.scaled(T=6, B=5, N=16)
    gb, gt = _scan_grads(sw, W.make_scan_inputs(sw), 0, sw.B)
    for r in range(world):
        got = np.load(tmp_path / f"rank{r}.npz")
        np.testing.assert_allclose(got["dsnn"], full, rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(got["gbeta"], gb, rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(got["gthr"], gt, rtol=1e-12, atol=1e-15)


class _FakeNet:
    """Stands in for DenseSNN on CPU: records the calls of a step."""

    def __init__(self, rank):
        self.calls = []
        self.rank = rank
        self.batch_total = None
        self.dW_flat = torch.full((4,), float(rank + 1))
        self.loss = torch.tensor([0.5 * (rank + 1)])

    def forward(self, X, labels, stream=None):
        self.calls.append(("forward", self.batch_total))

    def backward(self, X, stream=None):
        self.calls.append(("backward",))

    def update(self, stream=None):
        self.calls.append(("update", self.dW_flat.tolist(), float(self.loss)))


def _dp_rank_main(rank, world, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        net = _FakeNet(rank)
        dp = DataParallelDenseSNN(net, global_batch=128)
        dp.train_step(None, None)
        torch.save(net.calls, os.path.join(out_dir, f"calls{rank}.pt"))
    finally:
        dist.destroy_process_group()


def test_data_parallel_step_order(tmp_path):
    """Forward with the global-batch normaliser, backward, then the update
    sees dW and the loss already summed over both ranks."""
    world = 2
    mp.spawn(_dp_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True)
    for r in range(world):
        calls = torch.load(tmp_path / f"calls{r}.pt")
        assert calls[0] == ("forward", 128)
        assert calls[1] == ("backward",)
        assert calls[2] == ("update", [3.0] * 4, 1.5)


# ---------------------------------------------------------------------------
# The convolutional SNN: weight gradients, per-channel beta gradients, loss
# ---------------------------------------------------------------------------

def _csnn_problem():
    w = W.CSNN_C4.scaled(T=3, B=4, H=12, W=12, convs=((4, 5), (8, 3)), n_classes=5)
    inp = W.make_conv_inputs(w, seed=W.SEED_BASE + 78)
    convs = [c.float().numpy().astype(np.float64) * 3.0 for c in inp["convs"]]  # enough spikes
    Wfc = inp["Wfc"].float().numpy().astype(np.float64) * 3.0
    X = inp["X"].float().numpy().astype(np.float64)                             # [T, B, H, W, 1]
    y = inp["labels"].numpy().astype(np.int64)
    return w, convs, Wfc, X, y


def _csnn_grads(w, convs, Wfc, X, y, b0, b1, batch_total):
    """Oracle gradients (conv filters, readout, per-channel betas) and loss of
    samples [b0, b1), the loss averaged over batch_total samples."""
    nb = b1 - b0
    xb = X[:, b0:b1].reshape(w.T * nb, w.H, w.W, w.Cin)
    betas = [np.full(c, w.beta) for c, _ in w.convs]
    fwd = O.csnn_forward(xb, convs, Wfc, w.T, nb, betas, w.beta_fc, w.thr, reset=w.reset)
    res = O.csnn_backward(fwd, convs, Wfc, y[b0:b1], w.T, nb, betas, w.beta_fc, w.thr,
                          w.sg_param, reset=w.reset)
    k = nb / batch_total
    parts = [d.ravel() for d in res["dW"]] + [res["dW_fc"].ravel()] + \
        [d.ravel() for d in res["dbeta"]] + [[res["loss"]]]
    return np.concatenate(parts) * k


def _csnn_rank_main(rank, world, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        w, convs, Wfc, X, y = _csnn_problem()
        b0, b1 = shard_range(w.B, world, rank)
        flat = torch.tensor(_csnn_grads(w, convs, Wfc, X, y, b0, b1, w.B))
        allreduce_sum_([flat])
        np.save(os.path.join(out_dir, f"csnn{rank}.npy"), flat.numpy())
    finally:
        dist.destroy_process_group()


def test_csnn_sharded_gradients_sum_to_the_full_batch(tmp_path):
    """Two gloo ranks on halves of the batch: the summed filter, readout and
    per-channel beta gradients and the loss equal the full batch's."""
    world = 2
    mp.spawn(_csnn_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world,
             join=True)
    w, convs, Wfc, X, y = _csnn_problem()
    full = _csnn_grads(w, convs, Wfc, X, y, 0, w.B, w.B)
    assert np.abs(full[:-1]).max() > 1e-6
    for r in range(world):
        np.testing.assert_allclose(np.load(tmp_path / f"csnn{r}.npy"), full, rtol=1e-12,
                                   atol=1e-15)


class _FakeConvNet(_FakeNet):
    """Stands in for ConvSNN: also holds the betas' gradients."""

    def __init__(self, rank):
        super().__init__(rank)
        self.dbeta_flat = torch.full((2,), 10.0 * (rank + 1))

    def update(self, stream=None):
        self.calls.append(("update", self.dW_flat.tolist(), self.dbeta_flat.tolist(),
                           float(self.loss)))


def _dp_conv_rank_main(rank, world, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        from paper_2211_10725_gb300.data_parallel import DataParallelConvSNN
        net = _FakeConvNet(rank)
        DataParallelConvSNN(net, global_batch=256).train_step(None, None)
        torch.save(net.calls, os.path.join(out_dir, f"conv_calls{rank}.pt"))
    finally:
        dist.destroy_process_group()


def test_data_parallel_conv_step_sums_beta_gradients(tmp_path):
    """The convolutional network's step also sums the betas' gradients
    before the update."""
    world = 2
    mp.spawn(_dp_conv_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world,
             join=True)
    for r in range(world):
        calls = torch.load(tmp_path / f"conv_calls{r}.pt")
        assert calls[0] == ("forward", 256)
        assert calls[2] == ("update", [3.0] * 4, [30.0] * 2, 1.5)
