"""Model shape checks on the CPU: dc_model_weight_count follows the weight
order that include/drivecache.h documents, and dc_model_create rejects every
shape outside the documented support before it touches a device."""

import pytest

DTYPE_F32, DTYPE_BF16 = 0, 1
INVALID_ARG, UNSUPPORTED = 1, 6


@pytest.fixture(scope="module")
def dc():
    from paper_2608_16354_gb300 import _build, binding
    _build.build()
    binding.lib()
    return binding


def _desc(dc, **kw):
    f = dict(dtype=DTYPE_BF16, n_blocks=12, d_model=384, n_heads=6, mlp_ratio=4, channels=16,
             n_tokens=3584, n_poses=29, max_batch=16, max_steps=25)
    f.update(kw)
    m = dc.ModelDesc()
    for k, v in f.items():
        setattr(m, k, v)
    return m


def _documented_count(L, d, md, C, N, P):
    """The tensor list of the dc_model_create comment, summed."""
    stem = C * d + d + N * d + d * 256 + d + d * d + d + d * 3 * P + d
    ada = (6 * L + 2) * d * d + (6 * L + 2) * d
    block = 3 * d * d + 3 * d + d * d + d + md * d + md + d * md + d
    return stem + ada + L * block + C * d + C


@pytest.mark.parametrize("kw", [
    dict(), dict(n_blocks=2, d_model=1152, n_heads=16, n_tokens=14336, n_poses=61),
    dict(dtype=DTYPE_F32, n_blocks=2, d_model=64, n_heads=2, channels=4, n_tokens=128, n_poses=8),
    dict(dtype=DTYPE_F32, n_blocks=1, d_model=16, n_heads=2, mlp_ratio=3, channels=4, n_tokens=7,
         n_poses=1)])
def test_weight_count_follows_documented_order(dc, kw):
    m = _desc(dc, **kw)
    want = _documented_count(m.n_blocks, m.d_model, m.mlp_ratio * m.d_model, m.channels,
                             m.n_tokens, m.n_poses)
    assert dc.lib().dc_model_weight_count(dc.C.byref(m)) == want


@pytest.mark.parametrize("kw,status", [
    (dict(dtype=5), INVALID_ARG), (dict(n_blocks=0), INVALID_ARG), (dict(n_heads=5), INVALID_ARG),
    (dict(n_tokens=0), INVALID_ARG), (dict(max_steps=0), INVALID_ARG),
    (dict(channels=8), UNSUPPORTED), (dict(max_batch=65), UNSUPPORTED),
    (dict(d_model=3264, n_heads=51), UNSUPPORTED),             # d_model above 3072
    (dict(n_heads=12), UNSUPPORTED),                           # bf16 head dim 32
    (dict(d_model=320, n_heads=5), UNSUPPORTED),               # bf16 d_model % 192 != 0
    (dict(dtype=DTYPE_F32, d_model=384, n_heads=3), UNSUPPORTED),  # f32 head dim 128
    (dict(n_blocks=4097), UNSUPPORTED), (dict(mlp_ratio=17), UNSUPPORTED),
    (dict(n_tokens=(1 << 22) + 1, max_batch=1), UNSUPPORTED),
    (dict(n_tokens=1 << 21, max_batch=17), UNSUPPORTED),       # max_batch * n_tokens > 2^25
    (dict(n_poses=65537), UNSUPPORTED), (dict(max_steps=100001), UNSUPPORTED)])
def test_invalid_shapes_rejected_before_any_device_call(dc, kw, status):
    m = _desc(dc, **kw)
    assert dc.lib().dc_model_weight_count(dc.C.byref(m)) == 0
    blob = (dc.C.c_float * 4)()
    h = dc.C.c_void_p()
    got = dc.lib().dc_model_create(dc.C.byref(m), blob, 4, 0, dc.C.byref(h))
    assert got == status, dc.lib().dc_last_error().decode()
    assert not h.value


def test_weight_blob_size_is_checked_before_any_device_call(dc):
    m = _desc(dc, n_blocks=1)
    n = dc.lib().dc_model_weight_count(dc.C.byref(m))
    blob = (dc.C.c_float * 8)()
    h = dc.C.c_void_p()
    assert dc.lib().dc_model_create(dc.C.byref(m), blob, n - 1, 0, dc.C.byref(h)) == INVALID_ARG
    assert "expected" in dc.lib().dc_last_error().decode()


@pytest.mark.parametrize("args,status", [
    ((DTYPE_BF16, 0, 1, 1, 128, 64), INVALID_ARG),           # NULL qkv
    ((DTYPE_BF16, 16, 0, 1, 128, 64), INVALID_ARG),          # no slots
    ((DTYPE_BF16, 16, 1, 1, 128, 0), INVALID_ARG),           # head_dim 0
    ((DTYPE_BF16, 16, 256, 129, 128, 64), UNSUPPORTED),      # slots * heads > 2^15
    ((DTYPE_BF16, 16, 1, 1, (1 << 22) + 1, 64), UNSUPPORTED),
    ((DTYPE_BF16, 16, 1, 1, 128, 32), UNSUPPORTED),          # no bf16 kernel for dim 32
    ((DTYPE_F32, 16, 1, 1, 128, 128), UNSUPPORTED),          # no fp32 kernel for dim 128
    ((7, 16, 1, 1, 128, 64), INVALID_ARG)])                  # unknown dtype
def test_attention_arguments_checked_before_any_device_call(dc, args, status):
    dtype, qkv, slots, heads, n, dh = args
    # the pointers are never dereferenced: every case fails its checks first
    got = dc.lib().dc_attention(dtype, dc.C.c_void_p(qkv or None), slots, heads, n, dh,
                                dc.C.c_void_p(16), None)
    assert got == status, dc.lib().dc_last_error().decode()
