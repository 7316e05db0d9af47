"""GPU parity of the salient-bitmap conversions (Sec. 3.5 stores the salient set as a bitmap over the
input columns; qtea_gemv takes the ascending index list) against the oracle, bit for bit."""
import numpy as np
import pytest

import oracle
import synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def qt():
    import paper_2609_00224_gb300 as m
    m.load()
    return m


def random_bitmap(K, density, seed):
    """Words of random bits (bit b of word w = column 32 w + b), bits past K set too: they must be
    ignored."""
    rng = np.random.default_rng(seed)
    words = (K + 31) // 32
    bits = (rng.random((words, 32)) < density).astype(np.uint64)
    return (bits << np.arange(32, dtype=np.uint64)).sum(axis=1).astype(np.uint32)


KS = [1, 31, 32, 33, 1000, 4096, 14336, 40000, 100000]


@pytest.mark.parametrize("K", KS)
@pytest.mark.parametrize("density", [0.0, 0.03, 0.5, 1.0])
def test_bitmap_to_index_matches_oracle(qt, K, density):
    bm = random_bitmap(K, density, seed=K + int(density * 100))
    want = oracle.salient_from_bitmap(bm, K)
    dev = torch.from_numpy(bm.view(np.int32).copy()).cuda() if bm.size else torch.zeros(0, dtype=torch.int32).cuda()
    got = qt.qtea_salient_from_bitmap(dev, K)
    assert np.array_equal(got.cpu().numpy(), want)


@pytest.mark.parametrize("K", KS)
@pytest.mark.parametrize("density", [0.0, 0.03, 0.5, 1.0])
def test_index_to_bitmap_matches_oracle(qt, K, density):
    idx = oracle.salient_from_bitmap(random_bitmap(K, density, seed=7 * K + int(density * 10)), K)
    want = oracle.salient_to_bitmap(idx, K)
    got = qt.qtea_salient_to_bitmap(torch.from_numpy(idx).cuda() if idx.size else None, K)
    assert np.array_equal(got.cpu().numpy().view(np.uint32), want)


def test_bitmap_errors(qt):
    bm = torch.from_numpy(np.array([0x80000005, 0x81], np.uint32).view(np.int32)).cuda()
    with pytest.raises(qt.QteaError):
        qt.qtea_salient_from_bitmap(bm, 40, max_s=4)  # five columns marked
    assert qt.qtea_salient_from_bitmap(bm, 40, max_s=5).cpu().tolist() == [0, 2, 31, 32, 39]
    for bad in ([3, 3], [5, 2], [-1], [40]):
        with pytest.raises(qt.QteaError):
            qt.qtea_salient_to_bitmap(torch.tensor(bad, dtype=torch.int32).cuda(), 40)


def test_gemv_from_bitmap_is_identical(qt):
    """A problem whose salient set arrives as the paper's bitmap: converted on the device, the GEMV
    gives the same bits as with the index list."""
    p = synth.make_problem("bitmap", 1024, 4096, 1, 120, seed=11)
    bm = oracle.salient_to_bitmap(p.salient_idx, p.K)
    idx = qt.qtea_salient_from_bitmap(torch.from_numpy(bm.view(np.int32).copy()).cuda(), p.K)
    assert np.array_equal(idx.cpu().numpy(), p.salient_idx)
    f16 = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda().view(torch.float16)
    layout = qt.qtea_pack_layout(torch.from_numpy(p.T).cuda(), n_salient=p.s)
    args = (f16(p.x), layout, f16(p.alpha.reshape(-1)), f16(p.v))
    res = (f16(p.residual_vals), torch.from_numpy(p.residual_idx).cuda())
    y1 = qt.qtea_gemv(*args, torch.from_numpy(p.salient_idx).cuda(), *res)
    y2 = qt.qtea_gemv(*args, idx, *res)
    torch.cuda.synchronize()
    assert torch.equal(y1, y2)
