"""The datastore file (fc_datastore_save / fc_datastore_file_info /
fc_datastore_load), exercised on host arrays: no CUDA call is made, so this
runs without a GPU.  The stores are the oracle's own suffix arrays, bucket
tables and LCP arrays, and the on-disk layout is checked against its
definition (header fields, section order, the FNV-1a checksum recomputed
here from its published constants)."""
import os

import numpy as np
import pytest

fcm = pytest.importorskip("paper_2502_17139_gb300.fastcoder")


def store(orc, n, vocab, seed):
    rng = np.random.default_rng(seed)
    T = rng.integers(0, vocab, n).astype(np.uint32)
    if n > 100:
        T[n // 3:n // 3 + 40] = T[:40]
    sa = orc.suffix_array(T)
    return dict(tokens=T, sa=sa, bucket=orc.bucket(T, sa, vocab), lcp=orc.lcp(T, sa)), vocab


def fnv1a64_words(b: bytes) -> int:
    b = b + bytes(-len(b) % 8)
    h = 14695981039346656037
    for w in np.frombuffer(b, dtype="<u8").tolist():
        h = ((h ^ w) * 1099511628211) & 0xFFFFFFFFFFFFFFFF
    return h


@pytest.mark.parametrize("n,vocab,seed", [(1, 3, 0), (7, 2, 1), (5000, 30, 2), (70001, 300, 3)])
def test_round_trip_and_layout(orc, tmp_path, n, vocab, seed):
    ds, vocab = store(orc, n, vocab, seed)
    path = str(tmp_path / "ds.fcds")
    fcm.datastore_save_host(path, ds["tokens"], ds["sa"], ds["bucket"], ds["lcp"])
    assert fcm.fc_datastore_file_info(path) == (n, vocab)
    back = fcm.datastore_load_host(path)
    for k in ds:
        assert np.array_equal(back[k], ds[k]), k
    raw = open(path, "rb").read()
    assert raw[:8] == b"FCDSTORE"
    ver, voc = np.frombuffer(raw[8:16], "<u4").tolist()
    nn, pay, chk = np.frombuffer(raw[16:40], "<u8").tolist()
    assert (ver, voc, nn) == (1, vocab, n) and raw[40:64] == bytes(24)
    body = raw[64:]
    assert pay == len(body) == 9 * n + 4 * (vocab + 1)
    want = (ds["tokens"].astype("<u4").tobytes() + ds["sa"].astype("<u4").tobytes()
            + ds["bucket"].astype("<u4").tobytes() + ds["lcp"].tobytes())
    assert body == want
    assert chk == fnv1a64_words(body)


def test_rejects_damaged_files(orc, tmp_path):
    ds, vocab = store(orc, 3000, 17, 9)
    path = str(tmp_path / "ds.fcds")
    fcm.datastore_save_host(path, ds["tokens"], ds["sa"], ds["bucket"], ds["lcp"])
    good = open(path, "rb").read()

    def status_of(data, **kw):
        p = str(tmp_path / "bad.fcds")
        with open(p, "wb") as f:
            f.write(data)
        with pytest.raises(fcm.FastCoderError) as e:
            fcm.datastore_load_host(p)
        return e.value.status

    flipped = bytearray(good)
    flipped[64 + 4 * 3000 + 17] ^= 1          # one bit of the suffix array
    assert status_of(bytes(flipped)) == "FC_ERR_IO"
    assert status_of(good[:-1]) == "FC_ERR_IO"  # truncated
    assert status_of(good + b"\0") == "FC_ERR_IO"  # trailing bytes
    assert status_of(b"NOTASTORE" + good[9:]) == "FC_ERR_IO"
    with pytest.raises(fcm.FastCoderError) as e:
        fcm.fc_datastore_file_info(str(tmp_path / "missing.fcds"))
    assert e.value.status == "FC_ERR_IO"
    # buffers smaller than the file's store
    import ctypes as C
    small = np.empty(10, np.uint32)
    rc = fcm.LIB.fc_datastore_load(os.fsencode(path), small.ctypes.data, small.ctypes.data, small.ctypes.data,
                                   small.ctypes.data, 10, vocab, 1, None, None)
    assert fcm.STATUS[rc] == "FC_ERR_CAPACITY"
