"""Test helper: reads every section of an index file into numpy arrays (the
layout: a 256-byte header, then ten 256-byte-aligned sections W1, b1, W2, b2,
tau, bkt_off, cl_off, cent, ids, vec)."""
import struct

import numpy as np


def read_nrix(path):
    with open(path, "rb") as f:
        buf = f.read()
    assert buf[:8] == b"NRIXv001"
    _, dtype, N, D, H, b, K_max, t = struct.unpack_from("<IIQIIIII", buf, 8)
    n_cl, in_scale = struct.unpack_from("<Qf", buf, 48)
    offs = struct.unpack_from("<10Q", buf, 64)
    nb = (1 << b) + 1
    specs = [("W1", np.float32, H * D), ("b1", np.float32, H), ("W2", np.float32, b * H),
             ("b2", np.float32, b), ("tau", np.float32, b), ("bkt_off", np.uint32, nb),
             ("cl_off", np.uint32, n_cl + 1), ("cent", np.float32, n_cl * b),
             ("ids", np.uint32, N),
             ("vec", np.uint8 if dtype == 0 else np.float32, N * D)]
    out = dict(dtype=dtype, N=N, D=D, H=H, b=b, K_max=K_max, t=t, n_cl=n_cl, in_scale=in_scale)
    for (name, dt, n), o in zip(specs, offs):
        out[name] = np.frombuffer(buf, dtype=dt, count=n, offset=o)
    out["cent"] = out["cent"].reshape(n_cl, b)
    out["vec"] = out["vec"].reshape(N, D)
    return out
