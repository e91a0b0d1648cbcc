"""File tier of the version store (§3.5 metadata-driven recovery), host
side, no GPU: CRC-32C pinned by its published check value; the library's
CRC (sliced tables, pieces joined by polynomial arithmetic) against the
definition; and the library's manifest reader against directories the
independent writer in oracle/files.py makes -- with a torn tail, a record
damaged mid-log and a damaged block."""
import os

import numpy as np
import pytest

from oracle import files as F


def test_crc32c_check_value_and_forms():
    # the CRC catalogue's check value of CRC-32C (CRC-32/ISCSI) over "123456789"
    assert F.crc32c(b"123456789") == 0xE3069283
    assert F.crc32c_bitwise(b"123456789") == 0xE3069283
    rng = np.random.default_rng(0)
    for n in (0, 1, 3, 8, 9, 255, 1000):
        data = rng.integers(0, 256, n, dtype=np.uint8).tobytes()
        assert F.crc32c(data) == F.crc32c_bitwise(data)
    # continuation: the CRC of A then B equals the CRC of AB
    a, b = b"layer", b"check"
    assert F.crc32c(b, F.crc32c(a)) == F.crc32c(a + b)
    assert F.crc32c(b"") == 0


@pytest.fixture(scope="module")
def P():
    from paper_2609_27193_gb300 import build as B
    B.build()
    import paper_2609_27193_gb300 as P
    return P


def test_library_crc_matches_definition(P):
    rng = np.random.default_rng(1)
    for n in (0, 1, 7, 8, 9, 63, 64, 65, 4096, 65537):
        data = rng.integers(0, 256, n, dtype=np.uint8)
        assert P.crc32c(data) == F.crc32c(data.tobytes()), n
    assert P.crc32c(b"123456789") == 0xE3069283
    data = rng.integers(0, 256, 5000, dtype=np.uint8)
    assert P.crc32c(data[3000:], P.crc32c(data[:3000])) == F.crc32c(data.tobytes())


def test_library_crc_pieces_join():
    """Above 64 MiB the library splits the input over threads and joins the
    pieces' CRCs with x^(8n) products; chained 1 MiB calls (serial tables
    only) must give the same value."""
    import paper_2609_27193_gb300 as P
    rng = np.random.default_rng(2)
    n = (130 << 20) + 12345
    data = rng.integers(0, 256, n, dtype=np.uint8)
    whole = P.crc32c(data)
    crc = 0
    step = 1 << 20
    for a in range(0, n, step):
        crc = P.crc32c(data[a:a + step], crc)
    assert whole == crc


def _versions(rng, layer_bytes, steps):
    out = []
    for t in steps:
        for l, nb in enumerate(layer_bytes):
            if t == 0 or rng.random() < 0.5:
                out.append((l, t, rng.integers(0, 256, nb, dtype=np.uint8).tobytes()))
    return out


def test_manifest_read_matches_independent_writer(tmp_path, P):
    rng = np.random.default_rng(3)
    layer_bytes = [4096, 768, 12288, 256]
    vers = _versions(rng, layer_bytes, range(6))
    d = str(tmp_path / "ckpt")
    recs = F.write_dir(d, layer_bytes, vers)
    got, nl, lay, torn = P.manifest_read(d)
    assert nl == 4 and lay == F.layout_crc(layer_bytes) and not torn
    assert len(got) == len(recs)
    for g, r in zip(got, recs):
        for k in ("layer", "step", "offset", "bytes", "block_crc", "layout_crc"):
            assert g[k] == r[k], k
        assert g["intact"] == 1


def test_torn_tail_and_damaged_record_end_the_log(tmp_path, P):
    rng = np.random.default_rng(4)
    layer_bytes = [1024, 2048]
    vers = _versions(rng, layer_bytes, range(4))
    d = str(tmp_path / "ckpt")
    recs = F.write_dir(d, layer_bytes, vers)
    man = os.path.join(d, "manifest.lcm")
    with open(man, "ab") as f:                 # an append cut short
        f.write(F.record_bytes(0, 9, 0, 1024, 0, F.layout_crc(layer_bytes))[:37])
    got, _, _, torn = P.manifest_read(d)
    assert torn and len(got) == len(recs)
    assert F.read_dir(d)[3] and len(F.read_dir(d)[2]) == len(recs)
    raw = bytearray(open(man, "rb").read())
    k = 2                                      # damage record k: the log ends before it
    raw[F.REC * (1 + k) + 20] ^= 0x40
    open(man, "wb").write(bytes(raw))
    got, _, _, torn = P.manifest_read(d)
    assert torn and len(got) == k
    assert len(F.read_dir(d)[2]) == k


def test_damaged_block_is_not_intact(tmp_path, P):
    rng = np.random.default_rng(5)
    layer_bytes = [2048, 4096, 512]
    vers = _versions(rng, layer_bytes, range(5))
    d = str(tmp_path / "ckpt")
    recs = F.write_dir(d, layer_bytes, vers)
    bad = len(recs) - 2
    with open(os.path.join(d, "blocks.lcb"), "r+b") as f:
        f.seek(recs[bad]["offset"] + 17)
        b = f.read(1)
        f.seek(recs[bad]["offset"] + 17)
        f.write(bytes([b[0] ^ 1]))
    got, _, _, torn = P.manifest_read(d, verify_blocks=True)
    assert not torn
    assert [g["intact"] for g in got] == [int(i != bad) for i in range(len(recs))]
    _, _, orecs, _ = F.read_dir(d, verify_blocks=True)
    assert [int(r["intact"]) for r in orecs] == [g["intact"] for g in got]
    # the pick passes over the damaged version to the layer's next older one
    t_last = max(r["step"] for r in recs)
    pk = F.pick(orecs, layer_bytes, t_last)
    l = recs[bad]["layer"]
    older = [i for i, r in enumerate(recs) if r["layer"] == l and i != bad]
    assert pk[l] == max(older, key=lambda i: (recs[i]["step"], i))


def test_manifest_errors(tmp_path, P):
    with pytest.raises(P.LCError) as e:
        P.manifest_read(str(tmp_path / "missing"))
    assert e.value.status == 1
    d = tmp_path / "bad"
    d.mkdir()
    (d / "manifest.lcm").write_bytes(b"LCMH" + bytes(60))
    with pytest.raises(P.LCError) as e:
        P.manifest_read(str(d))
    assert e.value.status == 2


def test_record_beyond_the_block_file_is_not_intact(tmp_path, P):
    """A record whose CRC checks out but whose block lies past the end of a
    truncated block file is reported not intact, without reading it."""
    rng = np.random.default_rng(6)
    layer_bytes = [4096, 8192]
    vers = _versions(rng, layer_bytes, range(3))
    d = str(tmp_path / "ckpt")
    recs = F.write_dir(d, layer_bytes, vers)
    blocks = os.path.join(d, "blocks.lcb")
    with open(blocks, "r+b") as f:
        f.truncate(recs[-1]["offset"] + 100)
    got, _, _, torn = P.manifest_read(d, verify_blocks=True)
    assert not torn and len(got) == len(recs)
    assert [g["intact"] for g in got] == [1] * (len(recs) - 1) + [0]


def test_pick_matches_composite_rule_and_replay():
    """The record pick of recovery (§3.5, Eq. 8) against two other forms of
    the same rule.  The first is the C oracle's composite pick over the same
    versions, where an intact record of the right size and layout counts as
    durable.  The second is a replay that applies the valid records at or
    before t_fail in step order, record order breaking ties: each layer ends
    on its pick.  Random logs with ties, out-of-range layers, wrong sizes,
    foreign layouts and damaged blocks."""
    from oracle import oracle as O
    rng = np.random.default_rng(7)
    layer_bytes = [4096, 768, 12288, 256, 512]
    nl = len(layer_bytes)
    lay = F.layout_crc(layer_bytes)
    for _ in range(300):
        recs = []
        for _ in range(int(rng.integers(0, 40))):
            l = int(rng.integers(-1, nl + 1))
            in_range = 0 <= l < nl
            recs.append(dict(layer=l, step=int(rng.integers(0, 8)), offset=0,
                             bytes=layer_bytes[l] if in_range and rng.random() < 0.9 else 100,
                             block_crc=0, layout_crc=lay if rng.random() < 0.95 else lay ^ 1,
                             intact=bool(rng.random() < 0.85)))
        t_fail = int(rng.integers(-1, 9))
        pk = F.pick(recs, layer_bytes, t_fail)
        valid = [bool(r["intact"]) and 0 <= r["layer"] < nl and r["bytes"] == layer_bytes[r["layer"]]
                 and r["layout_crc"] == lay for r in recs]
        cp = O.composite_pick([r["layer"] for r in recs], [r["step"] for r in recs], valid, nl, t_fail)
        assert list(pk) == cp.tolist()
        state = [-1] * nl
        for i in sorted(range(len(recs)), key=lambda i: (recs[i]["step"], i)):
            if valid[i] and recs[i]["step"] <= t_fail:
                state[recs[i]["layer"]] = i
        assert list(pk) == state
