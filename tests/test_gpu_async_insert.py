"""Asynchronous inserts (lipcache_insert without a host count): the table's
size lives on the device, so batches chain on their stream without the host;
every call that needs the size settles it first (pytest -m gpu)."""
import numpy as np
import pytest

import oracle
import synth
from parity_utils import check_insert, check_probe

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    import __graft_entry__
    __graft_entry__.build()
    return torch.device("cuda", 0)


def T(x, dev):
    return torch.from_numpy(np.ascontiguousarray(x)).to(dev)


def make(dev, W, b, capacity, mode="conservative"):
    from paper_2608_13144_gb300.lipcache import LipCache
    c = LipCache(W.shape[1], W.shape[0], capacity, mode, device=dev)
    c.set_head(T(W, dev), T(b, dev))
    return c


@pytest.mark.parametrize("name,mode", [("cifar100", "conservative"), ("cifar100", "tight"), ("tiny", "conservative")])
def test_async_equals_sync(dev, name, mode):
    """Batches inserted without waiting give the same indices, radii and
    entries as the same batches inserted one synchronised call at a time; a
    probe afterwards (which settles the size) matches the oracle."""
    w = synth.WORKLOADS[name]
    W, b = synth.head(w)
    rows = synth.cache_rows(w)[:20000]
    Q, _ = synth.queries(w, rows)
    batch = 3000
    a = make(dev, W, b, len(rows), mode)
    s = make(dev, W, b, len(rows), mode)
    rd = T(rows, dev)
    outs_a, outs_s, n_s = [], [], 0
    for i in range(0, len(rows), batch):
        ia, ra, na = a.insert(rd[i:i + batch], wait=False)
        assert na is None
        outs_a.append((ia, ra))
        i_s, r_s, k = s.insert(rd[i:i + batch])
        outs_s.append((i_s, r_s))
        n_s += k
    assert a.size == s.size == n_s
    ia = np.concatenate([x[0].cpu().numpy() for x in outs_a])
    is_ = np.concatenate([x[0].cpu().numpy() for x in outs_s])
    ra = np.concatenate([x[1].cpu().numpy() for x in outs_a])
    rs = np.concatenate([x[1].cpu().numpy() for x in outs_s])
    assert np.array_equal(ia, is_) and np.array_equal(ra.view(np.uint32), rs.view(np.uint32))
    ea, es = a.entries(), s.entries()
    for k in ("keys", "radius", "label", "yG"):
        assert np.array_equal(ea[k], es[k]), k
    ref = oracle.build_cache(W, b, oracle.sigma_max(W), rows, radius_mode=int(mode == "tight"))
    head = ("tight", W, b, rows, 1.0) if mode == "tight" else (W, b, rows, 1.0)
    check_insert(ia, ra, n_s, ref, head)
    # a probe right after asynchronous inserts settles the size first
    a2 = make(dev, W, b, len(rows), mode)
    for i in range(0, len(rows), batch):
        a2.insert(rd[i:i + batch], wait=False)
    gi, gl, gd = [t.cpu().numpy() for t in a2.probe(T(Q[:1024], dev))]
    orc = oracle.probe(ref["keys"], ref["radius"], ref["label"], Q[:1024])
    check_probe(gi, gl, gd, ref, Q[:1024], orc)
    for c in (a, s, a2):
        assert c.info()["device_errors"] == 0
        c.close()


def test_async_capacity_and_mixed_calls(dev):
    """The capacity check counts unsettled rows as accepted and settles when
    that bound would be exceeded: with some rows rejected (payload != y^G
    under the consistency flag) a batch that fits the exact size is accepted,
    and a synchronised insert after asynchronous ones reports the right count
    and size."""
    w = synth.WORKLOADS["cifar10"].scaled(N=4000)
    W, b = synth.head(w)
    rows = synth.cache_rows(w)
    payload = np.zeros(len(rows), np.int32)  # class 0: most rows rejected
    cap = 2000
    c = make(dev, W, b, cap)
    rd, pd = T(rows, dev), T(payload, dev)
    c.insert(rd[:1000], pd[:1000], True, wait=False)
    c.insert(rd[1000:2000], pd[1000:2000], True, wait=False)  # bound 2000 = capacity
    idx, rad, n = c.insert(rd[2000:3000], pd[2000:3000], True)  # settles, then fits
    ref = oracle.build_cache(W, b, oracle.sigma_max(W), rows[:3000], payload=payload[:3000], require_consistency=True)
    assert c.size == len(ref["keys"]) <= cap
    assert n == int(ref["cert"]["accept"][2000:].sum())
    assert np.array_equal(idx.cpu().numpy(), ref["index"][2000:])
    e = c.entries()
    assert np.array_equal(e["keys"], ref["keys"].astype(np.float32))
    # filling to the exact capacity, then one row more is E_FULL
    from paper_2608_13144_gb300._lib import LipCacheError
    c2 = make(dev, W, b, 2000)
    c2.insert(rd[:1000], wait=False)
    c2.insert(rd[1000:2000], wait=False)
    with pytest.raises(LipCacheError) as err:
        c2.insert(rd[2000:2001], wait=False)
    assert err.value.status == 4 and c2.size == 2000  # every row of these heads is accepted
    c.close()
    c2.close()
