"""Checkpoint-directory format, written and read independently of the
library (TEST INFRASTRUCTURE ONLY; the product never imports this).

The file tier keeps every persisted layer version as a block in an
append-only block file and one fixed-size record per block in a manifest
(format in include/layercheck.h).  §3.5 recovery is metadata driven: the
records alone decide which version of each layer the composite at a failure
step uses (the newest at or before it, Eq. 8), and only those blocks are
read.  This module restates the format with Python's struct module and
CRC-32C from its definition, so that tests can write directories the
library must read (torn tails, damaged blocks) and read what the library
wrote.

CRC-32C: the Castagnoli polynomial x^32 + x^28 + x^27 + x^26 + x^25 + x^23
+ x^22 + x^20 + x^19 + x^18 + x^14 + x^13 + x^11 + x^10 + x^9 + x^8 + x^6 +
1, processed least significant bit first (reflected), with initial value and
final XOR 0xFFFFFFFF.  Pins: the published check value of CRC-32C, and the
byte-table form against the bit-serial form.
"""
import os
import struct

import numpy as np

# the polynomial's coefficients x^0 .. x^31, reflected into a 32-bit word
POLY_EXPONENTS = (0, 6, 8, 9, 10, 11, 13, 14, 18, 19, 20, 22, 23, 25, 26, 27, 28)
POLY_REFLECTED = sum(1 << (31 - e) for e in POLY_EXPONENTS)


def crc32c_bitwise(data, crc=0):
    """Bit-serial CRC-32C: one shift (and conditional reduction) per bit."""
    reg = crc ^ 0xFFFFFFFF
    for byte in bytes(data):
        reg ^= byte
        for _ in range(8):
            reg = (reg >> 1) ^ POLY_REFLECTED if reg & 1 else reg >> 1
    return reg ^ 0xFFFFFFFF


def _byte_table():
    t = []
    for b in range(256):
        r = b
        for _ in range(8):
            r = (r >> 1) ^ POLY_REFLECTED if r & 1 else r >> 1
        t.append(r)
    return t


_TABLE = _byte_table()


def crc32c(data, crc=0):
    """Byte-at-a-time CRC-32C with a 256-entry table."""
    reg = crc ^ 0xFFFFFFFF
    t = _TABLE
    for byte in bytes(data):
        reg = (reg >> 8) ^ t[(reg ^ byte) & 0xFF]
    return reg ^ 0xFFFFFFFF


HEADER_MAGIC = b"LCMH"
RECORD_MAGIC = b"LCVR"
FORMAT = 1
REC = 64
BLOCK_ALIGN = 4096


def layout_crc(layer_bytes):
    return crc32c(b"".join(struct.pack("<Q", int(b)) for b in layer_bytes))


def header_bytes(nlayers, layout):
    body = HEADER_MAGIC + struct.pack("<IiI", FORMAT, nlayers, layout) + bytes(44)
    return body + struct.pack("<I", crc32c(body))


def record_bytes(layer, step, offset, nbytes, block_crc, layout):
    body = RECORD_MAGIC + struct.pack("<iqQQII", layer, step, offset, nbytes, block_crc, layout) + bytes(20)
    assert len(body) == 60
    return body + struct.pack("<I", crc32c(body))


def write_dir(path, layer_bytes, versions, crc_of=crc32c):
    """A fresh directory holding `versions` = [(layer, step, block bytes)]
    in order, blocks on 4096-byte boundaries.  Returns the records."""
    os.makedirs(path, exist_ok=True)
    lay = layout_crc(layer_bytes)
    recs = []
    with open(os.path.join(path, "blocks.lcb"), "wb") as fb:
        off = 0
        for layer, step, block in versions:
            block = bytes(block)
            fb.seek(off)
            fb.write(block)
            recs.append(dict(layer=layer, step=step, offset=off, bytes=len(block),
                             block_crc=crc_of(block), layout_crc=lay))
            off = (off + len(block) + BLOCK_ALIGN - 1) // BLOCK_ALIGN * BLOCK_ALIGN
    with open(os.path.join(path, "manifest.lcm"), "wb") as fm:
        fm.write(header_bytes(len(layer_bytes), lay))
        for r in recs:
            fm.write(record_bytes(r["layer"], r["step"], r["offset"], r["bytes"], r["block_crc"],
                                  r["layout_crc"]))
    return recs


def read_dir(path, verify_blocks=False, crc_of=crc32c):
    """(nlayers, layout CRC, records, torn): the records up to the first
    short or invalid one.  With verify_blocks each record gets `intact`."""
    raw = open(os.path.join(path, "manifest.lcm"), "rb").read()
    head = raw[:REC]
    if len(head) < REC or head[:4] != HEADER_MAGIC or struct.unpack("<I", head[60:64])[0] != crc32c(head[:60]):
        raise ValueError("corrupt manifest header")
    fmt, nlayers, lay = struct.unpack("<IiI", head[4:16])
    if fmt != FORMAT:
        raise ValueError("unknown format %d" % fmt)
    recs = []
    off = REC
    while off + REC <= len(raw):
        r = raw[off:off + REC]
        if r[:4] != RECORD_MAGIC or struct.unpack("<I", r[60:64])[0] != crc32c(r[:60]):
            break
        layer, step, boff, nbytes, bcrc, rlay = struct.unpack("<iqQQII", r[4:40])
        recs.append(dict(layer=layer, step=step, offset=boff, bytes=nbytes, block_crc=bcrc,
                         layout_crc=rlay, intact=True))
        off += REC
    torn = off != len(raw)
    if verify_blocks and recs:
        with open(os.path.join(path, "blocks.lcb"), "rb") as fb:
            for r in recs:
                fb.seek(r["offset"])
                blk = fb.read(r["bytes"])
                r["intact"] = len(blk) == r["bytes"] and crc_of(blk) == r["block_crc"]
    return nlayers, lay, recs, torn


def read_block(path, rec):
    with open(os.path.join(path, "blocks.lcb"), "rb") as fb:
        fb.seek(rec["offset"])
        return np.frombuffer(fb.read(rec["bytes"]), dtype=np.uint8)


def pick(recs, layer_bytes, t_fail):
    """§3.5 / Eq. 8 over records: per layer, the index of the intact record
    of the right size with the largest step <= t_fail (the later record on
    a tie), or -1."""
    lay = layout_crc(layer_bytes)
    best = [-1] * len(layer_bytes)
    for i, r in enumerate(recs):
        l = r["layer"]
        if not (0 <= l < len(layer_bytes)) or r["step"] > t_fail or not r.get("intact", True):
            continue
        if r["bytes"] != layer_bytes[l] or r["layout_crc"] != lay:
            continue
        if best[l] < 0 or r["step"] >= recs[best[l]]["step"]:
            best[l] = i
    return best
