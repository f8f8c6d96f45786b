"""hf_fold (Eq. 9 folding of the Eq. 7 correction) against the oracle's
fold, and the transfer through GPU-folded maps against the oracle's
unfused path (y0 + (y0 B) G applied at transfer time)."""

import numpy as np
import pytest
import torch

from gpu_harness import Case, MAX_ABS_TOL, REL_FRO_TOL, MapFetcher, RowFetcher
from oracle import heterofold_oracle as O
from paper_2609_32259_gb300 import binding as B
from paper_2609_32259_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__ as g

    g.build()


def _factors(n_maps, d_R, rank, seed, dev, scale=0.5):
    g = torch.Generator(device="cpu").manual_seed(seed)
    Bm = torch.randn((n_maps, d_R, rank), generator=g) / np.sqrt(d_R)
    Gm = torch.randn((n_maps, rank, d_R), generator=g) * scale
    return Bm.to(dev), Gm.to(dev)


@pytest.mark.parametrize("dtype,in_place", [("bf16", False), ("bf16", True), ("f32", False)])
def test_fold_matches_oracle(dtype, in_place):
    dev = torch.device("cuda")
    n_maps, d_R, K, rank = 3, 256, 384, 16
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    g = torch.Generator(device="cpu").manual_seed(5)
    Wm = (torch.randn((n_maps, d_R, K), generator=g) / np.sqrt(K)).to(tdt).to(dev)
    b = (torch.randn((n_maps, d_R), generator=g) * 0.1).to(dev)
    Bm, Gm = _factors(n_maps, d_R, rank, 6, dev)
    W0 = Wm.double().cpu().numpy()
    b0 = b.double().cpu().numpy()
    Wf = Wm if in_place else torch.empty_like(Wm)
    bf = b if in_place else torch.empty_like(b)
    B.fold(dtype, Wm, b, Bm, Gm, Wf, bf)
    torch.cuda.synchronize()
    rel = 2.0 ** -8 if dtype == "bf16" else 1e-5
    for m in range(n_maps):
        Af, bref = O.fold(W0[m].T, b0[m], Bm[m].double().cpu().numpy(),
                          Gm[m].double().cpu().numpy())
        got = Wf[m].double().cpu().numpy()
        assert np.all(np.abs(got - Af.T) <= rel * np.abs(Af.T) + 1e-6), m
        assert np.allclose(bf[m].double().cpu().numpy(), bref, rtol=1e-5, atol=1e-6), m


def test_transfer_with_folded_maps_matches_unfused_oracle():
    w = W.llama_to_ministral(600).with_(L_s=4, L_r=3)
    c = Case(w)
    dev = c.dev
    n_maps = w.L_r * 2
    rank = 16
    W_orig = c.Wm.clone()
    b_orig = c.b.clone()
    Bm, Gm = _factors(n_maps, w.d_r, rank, 7, dev, scale=0.06)
    Wflat = c.Wm.view(n_maps, w.d_r, w.K)
    bflat = c.b.view(n_maps, w.d_r)
    B.fold("bf16", Wflat, bflat, Bm, Gm, Wflat, bflat)   # in place: the job's maps
    c.run()
    assert c.job.device_status() == 0
    Bn = Bm.double().cpu().numpy().reshape(w.L_r, 2, w.d_r, rank)
    Gn = Gm.double().cpu().numpy().reshape(w.L_r, 2, rank, w.d_r)
    ref = O.transfer_unfused(RowFetcher(c.sender), c.csr, c.segs, MapFetcher(W_orig),
                             b_orig.cpu().numpy(), c.r, Bn, Gn, H_r=w.H_r, D_r=w.D_r,
                             pos=c.pos, inv_freq_r=c.inv_freq_r)
    for (l, cc), y in ref.items():
        gpu = c.gpu_rows(l, cc, np.arange(c.tok.T_r))
        diff = gpu - y
        rel = float(np.linalg.norm(diff) / np.linalg.norm(y))
        assert rel <= REL_FRO_TOL and float(np.abs(diff).max()) <= MAX_ABS_TOL, (l, cc, rel)
    # the correction matters: the unfolded maps give a clearly different cache
    plain = O.transfer(RowFetcher(c.sender), c.csr, c.segs, MapFetcher(W_orig),
                       b_orig.cpu().numpy(), c.r, H_r=w.H_r, D_r=w.D_r, pos=c.pos,
                       inv_freq_r=c.inv_freq_r, layers=[0], roles=(1,))
    d = plain[(0, 1)] - ref[(0, 1)]
    assert np.linalg.norm(d) > 0.1 * np.linalg.norm(ref[(0, 1)])


def test_fold_ragged_tile_and_bad_arguments():
    dev = torch.device("cuda")
    g = torch.Generator(device="cpu").manual_seed(9)
    Wm = (torch.randn((2, 40, 70), generator=g) * 0.1).to(dev)   # K = 70: a ragged last tile
    b = torch.randn((2, 40), generator=g).to(dev)
    Bm, Gm = _factors(2, 40, 8, 10, dev)
    Wf = torch.empty_like(Wm)
    bf = torch.empty_like(b)
    B.fold("f32", Wm, b, Bm, Gm, Wf, bf)
    torch.cuda.synchronize()
    for m in range(2):
        Af, _ = O.fold(Wm[m].double().cpu().numpy().T, b[m].double().cpu().numpy(),
                       Bm[m].double().cpu().numpy(), Gm[m].double().cpu().numpy())
        assert np.allclose(Wf[m].double().cpu().numpy(), Af.T, rtol=1e-5, atol=1e-6)
    Bm6 = torch.zeros((2, 40, 6), device=dev)
    Gm6 = torch.zeros((2, 6, 40), device=dev)
    with pytest.raises(B.HFError) as e:
        B.fold("f32", Wm, b, Bm6, Gm6, Wf, bf)               # rank not a multiple of 4
    assert e.value.status == B.HF_ERR_UNSUPPORTED
