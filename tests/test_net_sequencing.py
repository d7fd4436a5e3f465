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
