"""Pins for the straight-through variant and the compressed 2:4 export of the oracle.

* Straight-through (Appendix, "Comparison with Straight-Through Gumbel-Top-K"):
  forward with the discrete mask, backward through the relaxation.  Pinned against
  torch.autograd (float64) of the usual straight-through construction
  mask = hard + S - stop_gradient(S), Wm = W * mask, on a plain restatement of the
  relaxation, and against the tau -> 0 limit of the soft forward.
* Compressed 2:4 export: a hand-worked golden row (tests/golden/), and the
  round trip to the dense pruned weights of the plain export.
"""
import json
import os

import numpy as np
import pytest

from oracle import roi_oracle as O
from workloads import bf16_bits, make_inputs

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "export_2of4_compressed.json")


def test_st_gradients_match_autograd_of_straight_through():
    torch = pytest.importorskip("torch")
    N, M, tau = 2, 4, 0.7
    W, phi, dWm = make_inputs(8, 64, "normal", 11)
    Wb, dWb = bf16_bits(W), bf16_bits(dWm)
    ph = phi.numpy()
    seed, step = 5, 3
    fwd = O.mask_fwd_st(ph, Wb, N, M, tau, seed, step)
    bwd = O.mask_bwd_st(ph, Wb, dWb, fwd["hard_bits"], N, M, tau, seed, step)
    # autograd of the straight-through construction on a plain restatement
    g = torch.tensor(O.gumbel_noise(seed, step, 0, 8, 64), dtype=torch.float64)
    phit = torch.tensor(ph.astype(np.float64).ravel(), requires_grad=True)
    Wt = torch.tensor(O.bf16_to_f32(Wb).astype(np.float64).ravel(), requires_grad=True)
    kappa = (phit + g).reshape(-1, M)
    alpha, S = kappa, torch.zeros_like(kappa)
    for _ in range(N):
        mu = torch.softmax(alpha / tau, dim=-1)
        S = S + mu
        alpha = alpha + torch.log(1 - mu)
    hard = torch.zeros_like(S)
    hard.scatter_(1, torch.topk(kappa.detach(), N, dim=-1).indices, 1.0)
    mask = hard + S - S.detach()
    Wm = Wt * mask.reshape(-1)
    (Wm * torch.tensor(O.bf16_to_f32(dWb).astype(np.float64).ravel())).sum().backward()
    assert np.array_equal(hard.numpy().astype(bool).ravel(), fwd["hard"].ravel())
    assert np.allclose(bwd["dlogits"].ravel(), phit.grad.numpy(), rtol=1e-9, atol=1e-15)
    # dW: the bf16 bits of dWm where kept, +0 elsewhere (autograd gives dWm * hard)
    assert np.array_equal(O.bf16_to_f32(bwd["dW"]).ravel(), Wt.grad.numpy().astype(np.float32))


def test_st_forward_is_the_small_tau_limit_of_the_soft_forward():
    W, phi, _ = make_inputs(6, 128, "normal", 4)
    Wb, ph = bf16_bits(W), phi.numpy()
    st = O.mask_fwd_st(ph, Wb, 2, 4, 1.0, 9, 1)
    soft = O.mask_fwd(ph, Wb, 2, 4, 1e-4, 9, 1)
    far = np.repeat(O.topn_key_gap(st["keys"].reshape(-1, 4), 2) > 1e-2, 4).reshape(6, 128)
    a = O.bf16_to_f32(st["Wm"])[far]
    b = O.bf16_to_f32(soft["Wm"])[far]
    assert far.mean() > 0.9 and np.array_equal(a, b)  # values (the soft side has -0 where W < 0)
    assert np.all(st["Wm"][~st["hard"]] == 0)          # +0 bits where pruned


def test_st_forward_keeps_exactly_n_weights_per_group():
    W, phi, _ = make_inputs(4, 96, "normal", 2)
    Wb = bf16_bits(W)
    for N, M in ((2, 4), (4, 8), (3, 8)):
        out = O.mask_fwd_st(phi.numpy(), Wb, N, M, 0.5, 1, 2)
        kept = (out["Wm"] == Wb).reshape(-1, M) & out["hard"].reshape(-1, M)
        assert np.all(kept.sum(-1) == N)


def test_compressed_export_golden_row():
    gold = json.load(open(GOLDEN))
    phi = np.array([[np.nan if x == "nan" else x for x in gold["logits"]]], dtype=np.float32)
    Wb = (0x3F80 + np.arange(32)).astype(np.uint16).reshape(1, 32)
    out = O.export_compressed_2of4(phi, Wb)
    assert [int(v) for v in out["values"].ravel()] == [int(x, 16) for x in gold["values_hex"]]
    assert [int(m) for m in out["meta"]] == [int(x, 16) for x in gold["meta_hex"]]


def test_compressed_export_round_trip_and_index_order():
    W, phi, _ = make_inputs(16, 256, "normal", 8)
    Wb = bf16_bits(W)
    phi = phi.numpy().copy()
    phi[0, :8] = 0.25          # ties
    phi[1, 4] = np.nan
    out = O.export_compressed_2of4(phi, Wb)
    dense = O.decompress_2of4(out["values"], out["meta"], 16, 256)
    assert np.array_equal(dense, O.hard_mask_export(phi, 2, 4, Wb)["W_pruned"])
    codes = (out["meta"][:, None] >> (4 * np.arange(8, dtype=np.uint32))) & 0xF
    assert np.all((codes & 3) < (codes >> 2))
