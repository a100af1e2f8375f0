"""Values the paper prints (tests/golden/, each file citing its table) against the library's and
the oracle's defaults and the synthetic workloads' shapes."""
import ctypes
import os

import pytest

from oracle.muon_ref import MuonParams
from oracle.soap_ref import HParams
from paper_2607_20548_gb300 import soap as S
from paper_2607_20548_gb300.workloads import WORKLOADS

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _pairs(name):
    out = {}
    for line in open(os.path.join(GOLDEN, name)):
        line = line.strip()
        if line and not line.startswith("#"):
            k, v = line.split()
            out[k] = float(v)
    return out


def test_soap_defaults_follow_the_kl_soap_table():
    """Every default of soap_default_hparams and of the oracle is the table's value, except beta1:
    the synthetic workloads step with beta1 = 0.95 (beta1 = beta2 = b); the table's 0.9 is one
    override away. The table's p = -1 is the inverse in the KL form (reading R2)."""
    t = _pairs("kl_soap_hparams.txt")
    hp = S.soap_hparams()
    S.load_library().soap_default_hparams(ctypes.byref(hp))
    assert hp.factor_beta == pytest.approx(t["beta_kron"])
    assert hp.beta2 == pytest.approx(t["beta2"])
    assert hp.eig_every == t["F"]
    assert hp.weight_decay == pytest.approx(t["weight_decay"])
    assert hp.eps == pytest.approx(t["eps"], rel=1e-6)
    assert t["beta1"] == 0.9 and hp.beta1 == pytest.approx(0.95)
    assert t["p"] == -1
    o = HParams()
    assert (o.factor_beta, o.beta2, o.eig_every, o.weight_decay, o.eps) == (
        t["beta_kron"], t["beta2"], t["F"], t["weight_decay"], t["eps"])


def test_muon_defaults_are_the_muon_table():
    t = _pairs("muon_hparams.txt")
    mh = S.muon_hparams()
    S.load_library().muon_default_hparams(ctypes.byref(mh))
    assert mh.beta1 == pytest.approx(t["beta1"])
    assert mh.weight_decay == pytest.approx(t["weight_decay"])
    assert mh.ns_steps == t["n"]
    assert mh.eps == pytest.approx(t["eps"], rel=1e-6)
    o = MuonParams()
    assert (o.beta1, o.weight_decay, o.eps) == (t["beta1"], t["weight_decay"], t["eps"])


def test_moe_workloads_use_the_qwen3_30b_a3b_widths():
    """The fine-grained MoE workloads take hidden 2048 and expert width 768 from the paper's
    Qwen3-30B-A3B row: every expert matrix is 2048 x 768 or 768 x 2048."""
    rows = {}
    for line in open(os.path.join(GOLDEN, "architectures.txt")):
        if line.strip() and not line.startswith("#"):
            name, hidden, layers, gqa, ffn = line.split()
            rows[name] = (int(hidden), int(layers), int(gqa), int(ffn))
    hidden, _, _, expert = rows["Qwen3-30B-A3B"]
    for name in ("moe_layer_64x768_h2048", "moe_stack_24x_h2048"):
        shapes = {(s.rows, s.cols) for s in WORKLOADS[name][0]}
        assert (hidden, expert) in shapes and (expert, hidden) in shapes
        assert all(hidden in sh for sh in shapes)
