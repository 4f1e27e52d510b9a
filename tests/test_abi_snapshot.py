"""Sampler-state snapshot format on the CPU: dc_snapshot_bytes follows the
layout that include/drivecache.h documents, and dc_snapshot_info accepts a
header built from that documentation and rejects every malformed one."""

import struct

import numpy as np
import pytest

DTYPE_F32, DTYPE_BF16 = 0, 1


@pytest.fixture(scope="module")
def dc():
    from paper_2608_16354_gb300 import _build, binding
    _build.build()
    binding.lib()
    return binding


def _desc(dc, dtype=DTYPE_BF16, N=3584, d=384, C=16):
    m = dc.ModelDesc()
    m.dtype, m.n_blocks, m.d_model, m.n_heads, m.mlp_ratio = dtype, 2, d, 6, 4
    m.channels, m.n_tokens, m.n_poses, m.max_batch, m.max_steps = C, N, 8, 16, 25
    return m


def _documented_size(B, K, cfg, N, d, C, elt):
    """The section sizes as the header comment lists them."""
    up = lambda x, a: (x + a - 1) // a * a
    host = 128 + 48 * B + 4 * up(B * (K + 1), 8) + 2 * 8 * B * (K + 1)
    payload = up(host, 256) + 2 * 4 * B * N * C
    Bi = 2 * B if cfg else B
    rows = up(payload, 256) + Bi * N * d * elt
    if elt == 2 and C == 16:  # the cache rows' sums (tensor-core interface)
        return up(rows, 256) + Bi * N * 2 * 4
    return rows


def _header(B, K, cfg, k_done, dtype, N, d, C, total, digest=0x0123456789ABCDEF, calls=7,
            magic=b"DCSNAP01", version=3):
    elt = 2 if dtype == DTYPE_BF16 else 4
    h = magic + struct.pack("<I8iIQQq", version, B, K, cfg, k_done, dtype, N, d, C, elt, digest,
                            total, calls)
    return h + bytes(128 - len(h))


@pytest.mark.parametrize("B,K,cfg,dtype,N,d,C", [
    (16, 25, 0, DTYPE_BF16, 3584, 384, 16), (16, 25, 1, DTYPE_BF16, 3584, 384, 16),
    (1, 10, 0, DTYPE_F32, 128, 64, 4), (3, 7, 1, DTYPE_F32, 77, 72, 16), (5, 1, 0, DTYPE_BF16, 1, 16, 1)])
def test_snapshot_bytes_follows_documented_layout(dc, B, K, cfg, dtype, N, d, C):
    elt = 2 if dtype == DTYPE_BF16 else 4
    got = dc.snapshot_bytes(_desc(dc, dtype, N, d, C), B, K, cfg)
    assert got == _documented_size(B, K, cfg, N, d, C, elt)


def test_snapshot_bytes_invalid_arguments(dc):
    m = _desc(dc)
    assert dc.snapshot_bytes(m, 0, 25) == 0
    assert dc.snapshot_bytes(m, 4, 0) == 0
    m.dtype = 7
    assert dc.snapshot_bytes(m, 4, 25) == 0


def _blob(B=2, K=6, cfg=1, k_done=3, dtype=DTYPE_F32, N=64, d=64, C=4, **kw):
    elt = 2 if dtype == DTYPE_BF16 else 4
    total = _documented_size(B, K, cfg, N, d, C, elt)
    h = _header(B, K, cfg, k_done, dtype, N, d, C, total, **kw)
    return np.frombuffer(h + bytes(total - 128), np.uint8).copy()


def test_snapshot_info_reads_documented_header(dc):
    info = dc.snapshot_info(_blob())
    assert info == dict(B=2, K=6, cfg=1, k_done=3, dtype=DTYPE_F32, n_tokens=64, d_model=64,
                        channels=4, digest=0x0123456789ABCDEF, backbone_calls=7)


@pytest.mark.parametrize("bad", [
    dict(magic=b"DCSNAP02"), dict(version=1), dict(version=2), dict(k_done=0), dict(k_done=7),
    dict(cfg=2), dict(B=0), dict(dtype=3), dict(calls=-1)])
def test_snapshot_info_rejects_malformed_headers(dc, bad):
    with pytest.raises(dc.DCError):
        dc.snapshot_info(_blob(**bad))


def test_snapshot_shapes_beyond_bounds_are_rejected(dc):
    """Shapes whose section sizes could overflow are refused by both calls."""
    m = _desc(dc)
    assert dc.snapshot_bytes(m, 1 << 17, 25) == 0
    assert dc.snapshot_bytes(m, 4, 200000) == 0
    m.n_tokens = 1 << 27
    assert dc.snapshot_bytes(m, 4, 25) == 0
    h = _header(B=1 << 20, K=4, cfg=0, k_done=2, dtype=DTYPE_F32, N=1 << 30, d=1 << 20, C=1 << 20,
                total=0)
    with pytest.raises(dc.DCError):
        dc.snapshot_info(np.frombuffer(h, np.uint8).copy())


def test_snapshot_info_rejects_wrong_sizes(dc):
    good = _blob()
    with pytest.raises(dc.DCError):
        dc.snapshot_info(good[:-1])  # truncated payload
    with pytest.raises(dc.DCError):
        dc.snapshot_info(np.concatenate([good, np.zeros(8, np.uint8)]))
    with pytest.raises(dc.DCError):
        dc.snapshot_info(good[:100])  # shorter than the header
    wrong = good.copy()  # the header's own size field disagrees with its shape
    wrong[56:64] = np.frombuffer(struct.pack("<Q", good.size + 8), np.uint8)
    with pytest.raises(dc.DCError):
        dc.snapshot_info(wrong)
