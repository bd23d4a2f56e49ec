"""Cross-quantizer transfer on the GPU against the oracle: the library's
distortion sweeps (one per quantizer family), fits and allocations give the
oracle's matrix J[a][b] = sum_i w_i D_i^b(b_i^a) on the same calibration
sample (Sec. 3.4 "Distortion calibration"; App. W Table 25)."""
import numpy as np
import pytest
import torch

from oracle import transfer as otr
from paper_2605_06675_gb300 import synth
from paper_2605_06675_gb300 import transfer as gtr
from paper_2605_06675_gb300.workloads import QWEN3_8B_8K

from .gpu_helpers import ensure_built, to_np

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("avg_bits,allowed", [(2.5, (2, 3, 4, 5, 6, 7, 8)), (3.0, (2, 3, 4, 8))])
def test_transfer_matrix_matches_oracle(avg_bits, allowed):
    ensure_built()
    wl = QWEN3_8B_8K.scaled(L=2, H_kv=4, allowed=allowed)
    dev = torch.device("cuda", 0)
    x = synth.calibration_sample(wl, T=128, device=dev)
    got = gtr.transfer_matrix(wl, dev, T=128, avg_bits=avg_bits, x=x)
    ref = otr.transfer_matrix(to_np(x), got["w"], avg_bits, wl.allowed_mask,
                              synth.hadamard_signs(wl.seed).numpy())
    assert got["names"] == ref["names"]
    for f in got["names"]:
        rel = np.abs(got["mse"][f] - ref["mse"][f]) / ref["mse"][f]
        assert rel.max() < 1e-5, (f, rel.max())
        np.testing.assert_allclose(got["beta"][f], ref["beta"][f], rtol=1e-5)
        same = np.mean(np.asarray(got["bits"][f]) == np.asarray(ref["bits"][f]))
        assert same >= 0.98, (f, same)     # near-ties may flip on 1e-5 MSE differences
    for a in got["names"]:
        for b in got["names"]:
            assert got["J"][a][b] == pytest.approx(ref["J"][a][b], rel=1e-4), (a, b)
        assert got["uniform"][a] == pytest.approx(ref["uniform"][a], rel=1e-5)
