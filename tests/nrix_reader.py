"""Test helper: reads every section of an index file into numpy arrays (the
layout: a 256-byte header, then ten 256-byte-aligned sections W1, b1, W2, b2,
tau, bkt_off, cl_off, cent, ids, vec)."""
import struct

import numpy as np


def read_nrix(path):
    with open(path, "rb") as f:
        buf = f.read()
    assert buf[:8] == b"NRIXv001"
    version, dtype, N, D, H, b, K_max, t = struct.unpack_from("<IIQIIIII", buf, 8)
    n_mid = struct.unpack_from("<I", buf, 152)[0] if version == 2 else 0
    mid_w = list(struct.unpack_from(f"<{n_mid}I", buf, 156)) if n_mid else []
    h_last = mid_w[-1] if mid_w else H
    n_cl, in_scale = struct.unpack_from("<Qf", buf, 48)
    offs = struct.unpack_from("<10Q", buf, 64)
    nb = (1 << b) + 1
    specs = [("W1", np.float32, H * D), ("b1", np.float32, H), ("W2", np.float32, b * h_last),
             ("b2", np.float32, b), ("tau", np.float32, b), ("bkt_off", np.uint32, nb),
             ("cl_off", np.uint32, n_cl + 1), ("cent", np.float32, n_cl * b),
             ("ids", np.uint32, N),
             ("vec", np.uint8 if dtype == 0 else np.float32, N * D)]
    out = dict(dtype=dtype, N=N, D=D, H=H, b=b, K_max=K_max, t=t, n_cl=n_cl, in_scale=in_scale,
               mid_w=mid_w)
    for (name, dt, n), o in zip(specs, offs):
        out[name] = np.frombuffer(buf, dtype=dt, count=n, offset=o)
    if n_mid:
        n = sum(w * p + w for w, p in zip(mid_w, [H] + mid_w[:-1]))
        out["mid"] = np.frombuffer(buf, dtype=np.float32, count=n,
                                   offset=struct.unpack_from("<Q", buf, 192)[0])
    out["cent"] = out["cent"].reshape(n_cl, b)
    out["vec"] = out["vec"].reshape(N, D)
    return out
