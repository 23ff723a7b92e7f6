"""Hand-built checkpoint files, byte by byte, for parser tests (no use of synth's encoder)."""
import struct


def entry(name, dtype, shape, offset, nbytes, name_bytes=None):
    nm = name.encode() if name_bytes is None else name_bytes
    return (struct.pack("<H", len(nm)) + nm + struct.pack("<BB", dtype, len(shape))
            + b"".join(struct.pack("<Q", s) for s in shape) + struct.pack("<QQ", offset, nbytes))


def assemble(entries, blobs, index_bytes=None, magic=b"WTCKPT01", n_entries=None, pad_to=None,
             extra_index=b""):
    """entries: raw entry bytes; blobs: list of (offset, bytes) written into the file image."""
    idx = struct.pack("<I", len(entries) if n_entries is None else n_entries) + b"".join(entries) + extra_index
    ib = len(idx) if index_bytes is None else index_bytes
    img = bytearray(magic + struct.pack("<Q", ib) + idx)
    end = max([len(img)] + [o + len(b) for o, b in blobs] + ([pad_to] if pad_to else []))
    img += b"\0" * (end - len(img))
    for o, b in blobs:
        img[o:o + len(b)] = b
    return bytes(img)


def header_len(entries):
    return 16 + 4 + sum(len(e) for e in entries)


def aligned(n, a=64):
    return -(-n // a) * a


def good_two_entry():
    """Two bf16 entries: 'a' [2,4] and 'b' [3] with known bytes."""
    e_a = entry("a", 1, (2, 4), 0, 16)
    e_b = entry("b", 1, (3,), 0, 6)
    o1 = aligned(header_len([e_a, e_b]))
    o2 = aligned(o1 + 16)
    e_a = entry("a", 1, (2, 4), o1, 16)
    e_b = entry("b", 1, (3,), o2, 6)
    blob_a = bytes(range(16))
    blob_b = bytes([0xAA, 0xBB, 0xCC, 0xDD, 0xEE, 0xFF])
    return assemble([e_a, e_b], [(o1, blob_a), (o2, blob_b)]), (o1, blob_a), (o2, blob_b)


def bad_files():
    """(label, file bytes) for every rejection rule of the container."""
    out = []
    good, (o1, ba), (o2, bb) = good_two_entry()
    out.append(("short", good[:10]))
    out.append(("magic", b"WTCKPT02" + good[8:]))
    hl = header_len([entry("a", 1, (2, 4), 0, 16)])
    # index length runs past the end of the file
    out.append(("index_past_eof", good[:8] + struct.pack("<Q", len(good)) + good[16:]))
    # index length smaller than the entries it holds
    e = entry("a", 1, (2, 4), 64, 16)
    out.append(("index_truncated", assemble([e], [(64, ba)], index_bytes=len(e))))
    # trailing junk inside the index
    e = entry("a", 1, (2, 4), 128, 16)
    out.append(("index_trailing", assemble([e], [(128, ba)], extra_index=b"\0" * 8)))
    # entry count larger than the index can hold
    out.append(("count_too_big", assemble([e], [(128, ba)], n_entries=1000)))
    off = aligned(hl)
    out.append(("dtype", assemble([entry("a", 9, (2, 4), off, 16)], [(off, ba)])))
    out.append(("ndim0", assemble([entry("a", 1, (), off, 2)], [(off, ba[:2])])))
    out.append(("ndim5", assemble([entry("a", 1, (1, 1, 1, 1, 8), off, 16)], [(off, ba)])))
    out.append(("nbytes", assemble([entry("a", 1, (2, 4), off, 18)], [(off, ba + b"\0\0")])))
    out.append(("misaligned", assemble([entry("a", 1, (2, 4), off + 16, 16)], [(off + 16, ba)])))
    out.append(("offset_in_index", assemble([entry("a", 1, (2, 4), 0, 16)], [], pad_to=64)))
    out.append(("blob_past_eof", assemble([entry("a", 1, (2, 4), off, 16)], [(off, ba[:8])])))
    e1 = entry("a", 1, (2, 4), 0, 16)
    e2 = entry("b", 1, (2, 4), 0, 16)
    o = aligned(header_len([e1, e2]))
    out.append(("overlap", assemble([entry("a", 1, (2, 4), o, 16), entry("b", 1, (2, 4), o, 16)],
                                    [(o, ba)], pad_to=o + 64)))
    out.append(("out_of_order", assemble([entry("a", 1, (2, 4), o + 64, 16), entry("b", 1, (2, 4), o, 16)],
                                         [(o, ba), (o + 64, ba)])))
    out.append(("duplicate_name", assemble([entry("a", 1, (2, 4), o, 16), entry("a", 1, (2, 4), o + 64, 16)],
                                           [(o, ba), (o + 64, ba)])))
    out.append(("empty_name", assemble([entry("", 1, (2, 4), off, 16)], [(off, ba)])))
    out.append(("nul_in_name", assemble([entry("", 1, (2, 4), off, 16, name_bytes=b"a\0b")], [(off, ba)])))
    big = (1 << 62, 1 << 3)
    out.append(("shape_overflow", assemble([entry("a", 1, big, off, 16)], [(off, ba)])))
    return out
