"""Host-side sequencing of the network training steps (no GPU needed): which
library launches each storage mode issues, in what order, and where the
forward ends.  The networks are built on the CPU with the one call that
needs a device (the scan workspace's initial write) replaced by a no-op;
no launch is issued."""
import pytest

from paper_2211_10725_gb300 import build_lib, snn
from paper_2211_10725_gb300 import workloads as W
from paper_2211_10725_gb300.csnn import ConvSNN
from paper_2211_10725_gb300.dsnn import DenseSNN


@pytest.fixture(autouse=True)
def host_only(monkeypatch):
    build_lib.build()
    monkeypatch.setattr(snn, "snn_workspace_init", lambda *a, **k: None)


def _names(net):
    return [n for n, _ in net.ops(None, None)]


DSNN_OPS = {
    "recompute": ["dense_fwd0", "scan_fwd0", "dense_fwd1", "scan_fwd1", "dense_fwd2", "scan_fwd2",
                  "ce_loss", "scan_bwd2", "dense_bwd2", "scan_bwd1", "dense_bwd1", "scan_bwd0",
                  "dense_bwd0", "adamw"],
    # the readout's trace is stored: its BPTT runs in the loss launch
    "mem": ["dense_fwd0", "scan_fwd0", "dense_fwd1", "scan_fwd1", "dense_fwd2", "scan_fwd2",
            "ce_loss", "dense_bwd2", "scan_bwd1", "dense_bwd1", "scan_bwd0", "dense_bwd0",
            "adamw"],
    # fused forward layers; the dX GEMMs of layers 2 and 1 carry the BPTT of
    # the layer below, so the dense backward computes dW only
    "fused": ["dense_scan_fwd0", "dense_scan_fwd1", "dense_scan_fwd2", "ce_loss", "dense_bwd2",
              "dense_scan_bwd2", "dense_bwd1", "dense_scan_bwd1", "dense_bwd0", "adamw"],
}


@pytest.mark.parametrize("save", sorted(DSNN_OPS))
def test_dense_network_launch_order(save):
    w = W.DSNN_C3
    net = DenseSNN(w, W.make_dense_inputs(w)["W"], device="cpu", save=save)
    names = _names(net)
    assert names == DSNN_OPS[save]
    # forward() runs up to and including the loss; backward() the rest but AdamW
    assert names[net._n_fwd() - 1] == "ce_loss"
    assert net.fused_loss == (save != "recompute")
    assert net.fused_bwd == (save == "fused")
    if save == "fused":
        assert all(i is None for i in net.I)   # the currents never exist
    else:
        assert all(i is not None for i in net.I)


def test_population_network_keeps_the_unfused_backward_at_one_step():
    w = W.DSNN_POP
    assert w.T == 1
    net = DenseSNN(w, W.make_dense_inputs(w)["W"], device="cpu", save="fused")
    assert not net.fused_bwd and net.fused_loss
    assert _names(net) == ["dense_scan_fwd0", "dense_scan_fwd1", "ce_loss", "dense_bwd1",
                           "scan_bwd0", "dense_bwd0", "adamw"]
    assert net.layers[-1].w.N == 504   # 10 classes x 50, padded to a multiple of 8


@pytest.mark.parametrize("save", ["recompute", "mem", "fused"])
def test_conv_network_launch_order(save):
    w = W.CSNN_C4
    inp = W.make_conv_inputs(w)
    net = ConvSNN(w, inp["convs"], inp["Wfc"], device="cpu", save=save)
    names = _names(net)
    assert names[net._n_fwd() - 1] == "ce_loss"
    assert names[-1] == "adamw"
    assert ("scan_bwd_out" in names) == (save == "recompute")
    assert net.fused_loss == (save != "recompute")
    if save == "fused":
        assert "conv_scan_fwd1" in names and "fc_scan_fwd" in names
        assert "scan_fwd1" not in names and "scan_fwd_out" not in names
    # the first layer is the direct few-channel convolution in every mode
    assert names[0] == "conv_fwd0" and "im2col0" not in names
    # every conv layer's reverse pass: pool backward, then scan, then conv
    for l in range(len(net.geo)):
        i = names.index(f"pool_bwd{l}")
        assert names[i + 1] == f"scan_bwd{l}" and names[i + 2] == f"conv_bwd{l}"


class _Recorder:
    """Stands in for the library calls of the reverse pass and for a
    snn.SideStream: records which product runs where, in call order."""

    def __init__(self, monkeypatch):
        self.log = []
        self.stream = "side"
        rec = self

        def dense_bwd(X, Wt, dI, dX, dW, ws, stream=None):
            rec.log.append(("dense_bwd", stream, dX is not None, dW is not None))

        monkeypatch.setattr(snn, "snn_dense_layer_bwd", dense_bwd)
        for name in ("snn_dense_leaky_bwd", "snn_rate_ce_leaky_bwd", "snn_rate_ce_loss",
                     "snn_adamw_step", "snn_leaky_bwd", "snn_maxpool2_bwd_nhwc",
                     "snn_col2im_nhwc", "snn_conv2d_small_dw_nhwc"):
            monkeypatch.setattr(snn, name, lambda *a, _n=name, **k: rec.log.append((_n,)))

    def fork(self, main, call):
        self.log.append(("fork",))
        call(self.stream)

    def join(self, main):
        self.log.append(("join",))


def test_dense_network_weight_gradients_on_the_side_stream(monkeypatch):
    """Fused mode: the upper layers' dW products are forked (queued on the
    side stream before the main stream's next product), the first layer's
    runs on the main stream and then joins the side stream, before AdamW."""
    w = W.DSNN_C3
    net = DenseSNN(w, W.make_dense_inputs(w)["W"], device="cpu", save="fused")
    rec = _Recorder(monkeypatch)
    ops = net.ops(None, None, None, rec)
    start = [n for n, _ in ops].index("dense_bwd2")
    for _, call in ops[start:-1]:   # the reverse pass, AdamW excluded
        call()
    log = rec.log
    assert log[0] == ("fork",) and log[1] == ("dense_bwd", "side", False, True)
    assert log[2] == ("snn_dense_leaky_bwd",)
    assert log[3] == ("fork",) and log[4] == ("dense_bwd", "side", False, True)
    assert log[5] == ("snn_dense_leaky_bwd",)
    assert log[6] == ("dense_bwd", None, False, True) and log[7] == ("join",)
    assert len(log) == 8


def test_dense_network_split_products_in_stored_mode(monkeypatch):
    """Stored-trace mode: each upper layer's dense backward forks its dW
    before issuing its dX on the main stream (which the next scan needs)."""
    w = W.DSNN_C3
    net = DenseSNN(w, W.make_dense_inputs(w)["W"], device="cpu", save="mem")
    rec = _Recorder(monkeypatch)
    ops = net.ops(None, None, None, rec)
    calls = dict(ops)
    calls["dense_bwd2"]()
    assert rec.log == [("fork",), ("dense_bwd", "side", False, True),
                       ("dense_bwd", None, True, False)]
    rec.log.clear()
    calls["dense_bwd0"]()
    assert rec.log == [("dense_bwd", None, False, True), ("join",)]


def test_conv_network_side_stream_forks_only_the_readout(monkeypatch):
    """CSNN: the readout's dW is forked; the second convolution's backward
    stays in line; the first layer's weight gradient joins the side
    stream."""
    w = W.CSNN_C4
    inp = W.make_conv_inputs(w)
    net = ConvSNN(w, inp["convs"], inp["Wfc"], device="cpu", save="fused")
    rec = _Recorder(monkeypatch)
    calls = dict(net.ops(None, None, None, rec))
    calls["fc_bwd"]()
    assert rec.log == [("fork",), ("dense_bwd", "side", False, True),
                       ("dense_bwd", None, True, False)]
    rec.log.clear()
    calls["conv_bwd1"]()
    assert rec.log == [("dense_bwd", None, True, True)]
    rec.log.clear()
    calls["conv_bwd0"]()
    assert rec.log == [("snn_conv2d_small_dw_nhwc",), ("join",)]
