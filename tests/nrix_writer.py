"""Test helper: writes an index file from explicit arrays, so tests can build
hand-made indexes (and malformed ones). Same layout the builder writes: a
256-byte header, then ten 256-byte-aligned sections
(W1, b1, W2, b2, tau, bkt_off, cl_off, cent, ids, vec); with hidden layers
after the first (mid: ((W, b), ...)), version 2 and an eleventh section
holding each such layer's W then b."""
import struct

import numpy as np


def write_nrix(path, vec, ids, bkt_off, cl_off, cent, tau, W1, b1, W2, b2, in_scale=1.0, K_max=0,
               t=0, truncate_to=None, mid=()):
    vec = np.ascontiguousarray(vec)
    dtype = 0 if vec.dtype == np.uint8 else 1
    N, D = vec.shape
    H = W1.shape[0]
    b = len(tau)
    n_cl = len(cl_off) - 1
    secs = [np.asarray(W1, np.float32), np.asarray(b1, np.float32), np.asarray(W2, np.float32),
            np.asarray(b2, np.float32), np.asarray(tau, np.float32),
            np.asarray(bkt_off, np.uint32), np.asarray(cl_off, np.uint32),
            np.asarray(cent, np.float32), np.asarray(ids, np.uint32), vec]
    if mid:
        secs.append(np.concatenate([np.concatenate([np.asarray(W, np.float32).ravel(),
                                                    np.asarray(bb, np.float32).ravel()])
                                    for W, bb in mid]))
    offs, cur = [], 256
    for s in secs:
        offs.append(cur)
        cur = (cur + s.nbytes + 255) & ~255
    hdr = bytearray(256)
    hdr[0:8] = b"NRIXv001"
    struct.pack_into("<IIQIIIIII", hdr, 8, 2 if mid else 1, dtype, N, D, H, b, K_max, t, 0)
    struct.pack_into("<Qf", hdr, 48, n_cl, in_scale)
    struct.pack_into("<10Q", hdr, 64, *offs[:10])
    struct.pack_into("<Q", hdr, 144, cur)
    if mid:
        struct.pack_into("<I", hdr, 152, len(mid))
        struct.pack_into(f"<{len(mid)}I", hdr, 156, *[np.asarray(W).shape[0] for W, _ in mid])
        struct.pack_into("<Q", hdr, 192, offs[10])
    buf = bytearray(cur)
    buf[0:256] = hdr
    for o, s in zip(offs, secs):
        buf[o:o + s.nbytes] = s.tobytes()
    if truncate_to is not None:
        buf = buf[:truncate_to]
    with open(path, "wb") as f:
        f.write(bytes(buf))
