"""Encoders with several hidden layers on the GPU (file version 2): the
library loads them, its encoder agrees with the oracle's double forward
(normwise 1e-2, the logit tolerance), searches fed the oracle's logits are
bit-exact, the GPU build writes the same bytes as the host builder (the
eleventh section included), save and extract keep the layers."""
import numpy as np
import pytest

import oracle
from gpu_util import need_cuda, recall
from nrix_reader import read_nrix
from test_oracle_mlp import B1, B2, M1, W1, W2, X

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def torch():
    return need_cuda()


def mlp_case(D=48, widths=(64, 32, 24, 16), b=12, n=20_000, seed=1):
    rng = np.random.default_rng(seed)
    centres = rng.normal(size=(64, D))
    base = centres[rng.integers(0, 64, n)] + 0.3 * rng.normal(size=(n, D))
    base = (base / np.linalg.norm(base, axis=1, keepdims=True)).astype(np.float32)
    q = centres[rng.integers(0, 64, 300)] + 0.3 * rng.normal(size=(300, D))
    q = (q / np.linalg.norm(q, axis=1, keepdims=True)).astype(np.float32)
    W1_ = (rng.normal(size=(widths[0], D)) / np.sqrt(D)).astype(np.float32)
    mid = tuple(((rng.normal(size=(w, p)) / np.sqrt(p)).astype(np.float32),
                 (0.01 * rng.normal(size=w)).astype(np.float32))
                for p, w in zip(widths[:-1], widths[1:]))
    W2_ = (rng.normal(size=(b, widths[-1])) / np.sqrt(widths[-1])).astype(np.float32)
    weights = (W1_, (0.01 * rng.normal(size=widths[0])).astype(np.float32), W2_,
               np.zeros(b, np.float32), mid)
    return base, q, weights, widths, b


# (D, hidden widths, b, rows): one hidden-layer chain per case; D = 272, 288,
# 512 and 1536 fp32 rows (1,088 to 6,144 bytes) take the long-row refinement
# with 4, 8 and 16 chunks a piece
# The tensor-core layer kernel takes D = 512, 1536 and 128 (every width a
# multiple of 64); the 704-wide layer has 176-column tiles (a 16-column
# remainder in the epilogue, accumulators wider than half of TMEM), and the
# uint8 case feeds its first layer through the producers' registers.
CASES = [("f32", 48, (64, 32, 24, 16), 12, 20_000), ("f32", 272, (128, 64), 12, 12_000),
         ("f32", 288, (128, 64), 12, 12_000), ("f32", 512, (256, 128, 64), 12, 12_000),
         ("f32", 1536, (512, 256, 128, 64), 16, 6_000), ("f32", 128, (704, 192), 20, 8_000),
         ("u8", 128, (256, 128), 16, 12_000)]


@pytest.fixture(scope="module", params=CASES, ids=[f"{c[0]}D{c[1]}" for c in CASES])
def built(torch, tmp_path_factory, request):
    from paper_2608_15438_gb300 import neuroute as nr
    from paper_2608_15438_gb300.builder import build_index, config

    dt, D, widths, b, n = request.param
    base, q, weights, widths, b = mlp_case(D, widths, b, n)
    if dt == "u8":  # the same points as bytes
        base = np.clip(np.rint(base * 400 + 128), 0, 255).astype(np.uint8)
        q = np.clip(np.rint(q * 400 + 128), 0, 255).astype(np.uint8)
    cfg = config(dt, base.shape[1], widths[0], b, 4, 16, mid=widths[1:])
    path = str(tmp_path_factory.mktemp("mlp") / "m.nrix")
    build_index(cfg, base, weights, path)
    return {"ix": nr.Index(path, 0), "orc": oracle.Index(path), "base": base, "q": q,
            "weights": weights, "cfg": cfg, "path": path}


def test_hand_worked_forward_on_the_gpu(torch, tmp_path):
    from nrix_writer import write_nrix
    from paper_2608_15438_gb300 import neuroute as nr

    m2 = (np.array([[-1, 1]], np.float32), np.zeros(1, np.float32))
    path = str(tmp_path / "h.nrix")
    write_nrix(path, np.zeros((1, 4), np.float32), [0], [0, 1, 1, 1, 1], [0, 1], np.zeros((1, 2)),
               np.zeros(2), np.pad(W1, ((0, 0), (0, 2))), B1, W2, B2, mid=(M1, m2))
    ix = nr.Index(path, 0)
    lg = ix.encode(torch.from_numpy(np.pad(X, ((0, 0), (0, 2)))).cuda())
    assert lg.cpu().numpy().tolist() == [[2.0, -2.0]]   # every step exact in fp32
    ix.close()


def test_encoder_within_tolerance(built, torch):
    lg = built["ix"].encode(torch.from_numpy(built["q"]).cuda()).cpu().numpy()
    ref = built["orc"].encode(built["q"])
    err = np.max(np.abs(lg - ref), axis=1)
    assert np.all(err <= 1e-2 * np.max(np.abs(ref), axis=1))


def test_search_bit_exact_and_recall(built, torch):
    ix, orc = built["ix"], built["orc"]
    q = built["q"]
    lg = orc.encode(q)
    kw = dict(t_low=4)
    ix.set_params(**kw)
    ids, d = ix.search_logits(torch.from_numpy(q).cuda(), torch.from_numpy(lg).cuda(), 10, 32, 64)
    st = ix.query_stats(len(q))
    torch.cuda.synchronize()
    ids_o, d_o, st_o = orc.search(q, 10, 32, 64, oracle.params(**kw), logits=lg)
    assert np.array_equal(ids.cpu().numpy(), ids_o)
    assert np.array_equal(d.cpu().numpy(), d_o)
    assert np.array_equal(st.cpu().numpy(), st_o)
    ids_e, _ = ix.search(torch.from_numpy(q).cuda(), 10, 32, 64)
    ids_oe, _, _ = orc.search(q, 10, 32, 64, oracle.params(**kw))
    truth = oracle.bruteforce(built["base"], q, 10)[0]
    assert abs(recall(ids_e.cpu().numpy(), truth) - recall(ids_oe, truth)) <= 0.002 + 1e-12
    ix.set_params()


def test_gpu_build_same_bytes_and_save_extract(built, torch, tmp_path):
    from paper_2608_15438_gb300 import neuroute as nr
    from paper_2608_15438_gb300.builder import build_index_from_logits, encode

    base, weights, cfg = built["base"], built["weights"], built["cfg"]
    logits = encode(cfg, base, weights)
    ph = str(tmp_path / "host.nrix")
    build_index_from_logits(cfg, base, logits, weights, ph)
    bd = nr.Builder(cfg, base.shape[0], weights, 0)
    bd.set_logits(torch.from_numpy(logits).cuda(), 0)
    torch.cuda.synchronize()
    bd.finish()
    bd.place(torch.from_numpy(base).cuda(), 0)
    ix = bd.end()
    pg = str(tmp_path / "gpu.nrix")
    ix.save(pg)
    assert open(ph, "rb").read() == open(pg, "rb").read()
    f = read_nrix(pg)
    assert f["mid_w"] == list(cfg.mid_w[: cfg.n_mid])
    # extract keeps the layers; the oracle on it answers like the whole index
    codes, nprobe = ix.route(torch.from_numpy(built["orc"].encode(built["q"][:20])).cuda(), 8)
    c = codes.cpu().numpy().view(np.uint32)
    used = np.concatenate([c[i, :n] for i, n in enumerate(nprobe.cpu().numpy())])
    sub = str(tmp_path / "sub.nrix")
    ix.extract(used, sub)
    assert read_nrix(sub)["mid_w"] == f["mid_w"]
    assert np.array_equal(read_nrix(sub)["mid"], f["mid"])
    # a GPU-encoded build of the same rows gives logits within tolerance
    bd = nr.Builder(cfg, base.shape[0], weights, 0)
    bd.encode(torch.from_numpy(base).cuda(), 0)
    torch.cuda.synchronize()
    bd.finish()
    bd.place(torch.from_numpy(base).cuda(), 0)
    ix2 = bd.end()
    tau = ix2.thresholds()
    assert np.allclose(tau, np.sort(logits, axis=0)[(base.shape[0] - 1) // 2], atol=1e-3)
    ix.close()
    ix2.close()


def test_layer_kernel_wait_expiry_is_flagged(built, torch):
    """The per-layer tensor-core encoder (D and every hidden width multiples
    of 64) under wait_limit_us < 0: every hand-off wait not complete when
    first tested gives up, the kernel waits for its bulk copies and MMAs in
    flight, frees its tensor memory and sets the device flag
    (NR_ERR_DEVICE_CHECK); the next encode on the same context is right."""
    from paper_2608_15438_gb300 import neuroute as nr

    ix, cfg = built["ix"], built["cfg"]
    if cfg.D % 64 or cfg.H % 64 or any(w % 64 for w in cfg.mid_w[: cfg.n_mid]):
        pytest.skip("shape of the CUDA-core encoder")
    q = torch.from_numpy(built["q"]).cuda()
    ix.set_params(wait_limit_us=-1)
    try:
        ix.encode(q)
        torch.cuda.synchronize()
        with pytest.raises(nr.NRError) as e:
            ix.last_stats()
        assert e.value.status == -6  # NR_ERR_DEVICE_CHECK
    finally:
        ix.set_params()
    ix.last_stats()
    lg = ix.encode(q).cpu().numpy()
    ref = built["orc"].encode(built["q"])
    assert np.all(np.abs(lg - ref).max(1) <= 1e-2 * np.abs(ref).max(1))


def test_encoder_across_row_blocks(built, torch):
    """A batch longer than the layer-by-layer encoder's row block (2^18 rows,
    the unit its activation scratch holds): rows on both sides of the block
    boundary and in the ragged last tile agree with the oracle's forward."""
    cfg = built["cfg"]
    if cfg.D % 64 or cfg.H % 64 or any(w % 64 for w in cfg.mid_w[: cfg.n_mid]):
        pytest.skip("shape of the CUDA-core encoder")
    n = (1 << 18) + 1000 + 37
    rng = np.random.default_rng(5)
    q = built["q"]
    if q.dtype == np.uint8:
        x = np.clip(q[rng.integers(0, len(q), n)].astype(np.int16) + rng.integers(-3, 4, (n, q.shape[1])),
                    0, 255).astype(np.uint8)
    else:
        x = q[rng.integers(0, len(q), n)] + 0.05 * rng.normal(size=(n, q.shape[1])).astype(np.float32)
    lg = built["ix"].encode(torch.from_numpy(x).cuda()).cpu().numpy()
    pick = np.r_[0:64, (1 << 18) - 64:(1 << 18) + 64, n - 101:n]
    ref = built["orc"].encode(x[pick])
    err = np.max(np.abs(lg[pick] - ref), axis=1)
    assert np.all(err <= 1e-2 * np.max(np.abs(ref), axis=1))


def test_encoder_misaligned_input(built, torch):
    """Input rows that do not start on a 16-byte boundary take the CUDA-core
    encoder (the tensor-core kernels copy 16-byte pieces); the logits agree
    with the oracle's within the same tolerance."""
    q = built["q"]
    n, D = q.shape
    esz = q.dtype.itemsize
    tdt = torch.uint8 if q.dtype == np.uint8 else torch.float32
    buf = torch.zeros(n * D + 16 // esz, dtype=tdt, device="cuda")
    off = 4 // esz if esz < 4 else 1           # 4 bytes past a 16-byte boundary
    x = buf[off:off + n * D].view(n, D)
    x.copy_(torch.from_numpy(q).cuda())
    assert x.data_ptr() % 16 != 0
    lg = built["ix"].encode(x).cpu().numpy()
    ref = built["orc"].encode(q)
    err = np.max(np.abs(lg - ref), axis=1)
    assert np.all(err <= 1e-2 * np.max(np.abs(ref), axis=1))


@pytest.mark.parametrize("n", [1, 5, 127, 129])
def test_encoder_small_batches(built, torch, n):
    """Batches smaller than one 128-row tile (and one row past it): the tile's
    missing rows are zeros on the way in and are not written out."""
    q = built["q"][:n]
    lg = built["ix"].encode(torch.from_numpy(np.ascontiguousarray(q)).cuda()).cpu().numpy()
    ref = built["orc"].encode(q)
    assert lg.shape == ref.shape
    err = np.max(np.abs(lg - ref), axis=1)
    assert np.all(err <= 1e-2 * np.max(np.abs(ref), axis=1))
