"""Cross-quantizer transfer on the GPU against the oracle (Sec. 3.4
"Distortion calibration"; App. W Table 25). The library's distortion sweep of
every quantizer family matches the oracle's sweep on the same calibration
sample within the sweep tolerance; on the library's own MSE the oracle's fit
and allocation give the library's bits exactly, and the matrix
J[a][b] = sum_i w_i D_i^b(b_i^a) equals the oracle's composition."""
import numpy as np
import pytest
import torch

from oracle import alloc as oalloc
from oracle import calib as ocalib
from oracle import transfer as otr
from paper_2605_06675_gb300 import synth
from paper_2605_06675_gb300 import transfer as gtr
from paper_2605_06675_gb300.workloads import QWEN3_8B_8K

from .gpu_helpers import ensure_built, to_np
from .test_gpu_parity import MSE_RTOL

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("avg_bits,allowed", [(2.5, (2, 3, 4, 5, 6, 7, 8)), (3.0, (2, 3, 4, 8))])
def test_transfer_matrix_matches_oracle(avg_bits, allowed):
    ensure_built()
    wl = QWEN3_8B_8K.scaled(L=2, H_kv=4, allowed=allowed)
    dev = torch.device("cuda", 0)
    x = synth.calibration_sample(wl, T=128, device=dev)
    got = gtr.transfer_matrix(wl, dev, T=128, avg_bits=avg_bits, x=x)
    names = got["names"]
    assert names == list(otr.FAMILIES)
    signs = synth.hadamard_signs(wl.seed).numpy()
    w = got["w"]
    n = x.shape[0]
    for f in names:
        # the sweep: the oracle's own MSE on the same sample, within the
        # sweep tolerance (fp32 group sums against exact fp64 squares)
        ref_mse, _, _ = otr.family_model(to_np(x), f, signs)
        rel = np.abs(got["mse"][f] - ref_mse) / ref_mse
        assert rel.max() < MSE_RTOL, (f, rel.max())
        # fit + allocation on the library's MSE: bit-identical to the oracle
        oa, ob, _ = ocalib.fit_distortion(got["mse"][f], 2, 6, 0.96, np.arange(n) % 2)
        np.testing.assert_array_equal(got["alpha"][f], oa)
        np.testing.assert_array_equal(got["beta"][f], ob)
        obits, _ = oalloc.allocate(w, oa, ob, avg_bits, wl.allowed_mask)
        assert list(got["bits"][f]) == list(obits), f
    # the matrix: the oracle's weighted distortion of every allocation on
    # every family's (library) MSE
    for a in names:
        for b in names:
            ref = otr.weighted_distortion(w, got["mse"][b], got["bits"][a])
            assert got["J"][a][b] == pytest.approx(ref, rel=1e-12), (a, b)
        ref_u = otr.weighted_distortion(w, got["mse"][a], otr.uniform_bits(n, avg_bits))
        assert got["uniform"][a] == pytest.approx(ref_u, rel=1e-12)
