"""Host-side argument checks of the C ABI, on the CPU.

Every entry point validates its arguments before it touches the device: a
null pointer, a negative size, t < 1, a coefficient outside its range or an
unknown dtype returns BOM_EINVAL; an unaligned buffer or a size beyond a
kernel's limit returns BOM_ENOTSUP; an empty range (n = 0) is a no-op that
returns BOM_OK without reading any pointer.  None of these calls dereferences
a pointer or starts a CUDA context, so they run without a GPU; the stream is
passed as 0 so that the binding does not ask torch for one.
"""
import pytest

from paper_2609_36738_gb300 import bom as B

ALIGNED = 0x10000          # fake device addresses: never dereferenced by these calls
UNALIGNED = 0x10004


@pytest.fixture(scope="module")
def built():
    from paper_2609_36738_gb300 import build
    build.build()
    return B.lib()


def _code(fn, *args, **kw):
    try:
        fn(*args, **kw)
    except B.BomError as e:
        return e.code
    return B.BOM_OK


def _upd(**over):
    a = dict(theta=ALIGNED, g=ALIGNED, g_dtype=B.BOM_F32, hvec=None, v=ALIGNED, theta_bf16=None, n=1024,
             lr=1e-3, wd=0.1, lam=0.5, beta2=0.999, eps=1e-8, t=1, stream=0)
    a.update(over)
    return a


@pytest.mark.parametrize("over, code", [
    (dict(n=-1), "BOM_EINVAL"),
    (dict(t=0), "BOM_EINVAL"),
    (dict(theta=None), "BOM_EINVAL"),
    (dict(g=None), "BOM_EINVAL"),
    (dict(v=None), "BOM_EINVAL"),
    (dict(g_dtype=7), "BOM_EINVAL"),
    (dict(beta2=1.0), "BOM_EINVAL"),
    (dict(beta2=-0.1), "BOM_EINVAL"),
    (dict(beta2=float("nan")), "BOM_EINVAL"),
    (dict(eps=-1e-8), "BOM_EINVAL"),
    (dict(theta=UNALIGNED), "BOM_ENOTSUP"),
    (dict(g=UNALIGNED), "BOM_ENOTSUP"),
    (dict(hvec=UNALIGNED), "BOM_ENOTSUP"),
    (dict(theta_bf16=UNALIGNED), "BOM_ENOTSUP"),
    (dict(n=0, theta=None, g=None, v=None), "BOM_OK"),
])
def test_bom_update_checks(built, over, code):
    assert _code(B.bom_update, **_upd(**over)) == getattr(B, code)


@pytest.mark.parametrize("over, code", [
    (dict(max_norm=0.0), "BOM_EINVAL"),
    (dict(max_norm=float("nan")), "BOM_EINVAL"),
    (dict(sq=None), "BOM_EINVAL"),
    (dict(t=0), "BOM_EINVAL"),
    (dict(v=UNALIGNED), "BOM_ENOTSUP"),
    (dict(n=0, theta=None, g=None, v=None), "BOM_OK"),
])
def test_bom_update_clipped_checks(built, over, code):
    a = _upd(sq=ALIGNED, max_norm=1.0)
    a.update(over)
    assert _code(B.bom_update_clipped, **a) == getattr(B, code)


@pytest.mark.parametrize("over, code", [
    (dict(block=0), "BOM_EINVAL"),
    (dict(v_blocks=None), "BOM_EINVAL"),
    (dict(g_dtype=-1), "BOM_EINVAL"),
    (dict(eps=float("nan")), "BOM_EINVAL"),
    (dict(g=UNALIGNED), "BOM_ENOTSUP"),
    (dict(n=0, theta=None, g=None, v_blocks=None), "BOM_OK"),
])
def test_bom_update_blockshared_checks(built, over, code):
    a = _upd(block=128)
    a["v_blocks"] = a.pop("v")
    a.update(over)
    assert _code(B.bom_update_blockshared, **a) == getattr(B, code)


@pytest.mark.parametrize("over, code", [
    (dict(M=0), "BOM_EINVAL"),
    (dict(N=0), "BOM_EINVAL"),
    (dict(K=-1), "BOM_EINVAL"),
    (dict(A=None), "BOM_EINVAL"),
    (dict(D=None), "BOM_EINVAL"),
    (dict(ldd=130), "BOM_ENOTSUP"),         # fp32 output rows must start on 16 bytes
    (dict(ldd=64), "BOM_ENOTSUP"),          # ldd < N
    (dict(D=UNALIGNED), "BOM_ENOTSUP"),
])
def test_bom_gemm_bf16_checks(built, over, code):
    a = dict(A=ALIGNED, lda=256, a_mn_major=False, B=ALIGNED, ldb=256, b_mn_major=False, D=ALIGNED, ldd=128,
             M=128, N=128, K=256, alpha=1.0, stream=0)
    a.update(over)
    assert _code(B.bom_gemm_bf16, **a) == getattr(B, code)


@pytest.mark.parametrize("over, code", [
    (dict(n_rows=0), "BOM_EINVAL"),
    (dict(n_cols=0), "BOM_EINVAL"),
    (dict(ldx=32), "BOM_EINVAL"),           # ldx < n_cols
    (dict(x=None), "BOM_EINVAL"),
    (dict(out=None), "BOM_EINVAL"),
    (dict(dtype=9), "BOM_EINVAL"),
    (dict(x=UNALIGNED), "BOM_ENOTSUP"),
    # ceil(n_rows / 128) * n_cols above the fixed 2^20-float scratch
    (dict(n_rows=129, n_cols=(1 << 19) + 8, ldx=(1 << 19) + 8), "BOM_ENOTSUP"),
    # more than 65,535 row ranges of 128 rows, with few columns
    (dict(n_rows=128 * 65535 + 1, n_cols=8, ldx=8), "BOM_ENOTSUP"),
    # sizes whose product would overflow 64 bits are refused, not wrapped
    (dict(n_rows=1 << 40, n_cols=(1 << 62) + 1, ldx=(1 << 62) + 1), "BOM_ENOTSUP"),
    (dict(n_rows=(1 << 62) + 1, n_cols=8, ldx=8), "BOM_ENOTSUP"),
])
def test_bom_colsum_noalloc_checks(built, over, code):
    a = dict(x=ALIGNED, dtype=B.BOM_BF16, ldx=64, n_rows=256, n_cols=64, weights=None, out=ALIGNED, stream=0)
    a.update(over)
    assert _code(B.bom_colsum_noalloc, **a) == getattr(B, code)


def test_null_handles_are_rejected(built):
    assert _code(B.bom_step, None, ALIGNED, ALIGNED, 8, [ALIGNED], ALIGNED, 1, [ALIGNED], stream=0) == B.BOM_EINVAL
    assert _code(B.bom_get_stats, None, stream=0) == B.BOM_EINVAL
    assert _code(B.bom_graph_launch, None, stream=0) == B.BOM_EINVAL
    assert _code(B.bom_sqnorm, None, ALIGNED, B.BOM_BF16, None, 0.5, 16, ALIGNED, stream=0) == B.BOM_EINVAL
    assert _code(B.bom_own_step_moment, None, ALIGNED, ALIGNED, ALIGNED, ALIGNED, 16, 0.9, 1, stream=0) == B.BOM_EINVAL
    assert _code(B.bom_trace, None, True) == B.BOM_EINVAL


def test_grid_row_limits_are_refused_at_init(built):
    """Per-row passes put 64-row blocks on gridDim.y (at most 65,535), so
    max_rows above 4,194,240 is refused when the handle is made, as is an fp32
    output width above the same bound (its weight-gradient GEMM has M = that
    width); the bf16 path takes any vocabulary up to 2^30."""
    lim = 64 * 65535
    lin = [(B.BOM_LAYER_LINEAR_GELU, 1, 64, 128)]
    assert B.bom_workspace_bytes(B.make_config(lim, 64, 10, lin, True, B.BOM_F32)) > 0
    assert B.bom_workspace_bytes(B.make_config(lim + 1, 64, 10, lin, True, B.BOM_F32)) == -1
    assert B.bom_workspace_bytes(B.make_config(lim + 1, 64, 10, [], False, B.BOM_BF16)) == -1
    assert B.bom_workspace_bytes(B.make_config(16, 64, lim, lin, True, B.BOM_F32)) > 0
    assert B.bom_workspace_bytes(B.make_config(16, 64, lim + 1, lin, True, B.BOM_F32)) == -1
    wide = [(B.BOM_LAYER_LINEAR_GELU, 1, 64, lim + 1)]
    assert B.bom_workspace_bytes(B.make_config(16, 64, 10, wide, True, B.BOM_F32)) == -1
    assert B.bom_workspace_bytes(B.make_config(16, 64, lim + 1, [], False, B.BOM_BF16)) > 0


def test_binding_fails_loudly_without_the_library(tmp_path, monkeypatch):
    """There is no CPU fallback: with libbom.so absent, loading the library and
    every compute entry point raise instead of computing anything."""
    monkeypatch.setattr(B, "LIB_PATH", str(tmp_path / "libbom.so"))
    monkeypatch.setattr(B, "_LIB", None)
    with pytest.raises(RuntimeError, match="missing"):
        B.lib()
    with pytest.raises(RuntimeError, match="missing"):
        B.bom_update(**_upd())
    with pytest.raises(RuntimeError, match="missing"):
        B.bom_workspace_bytes(B.make_config(16, 64, 10, [], False, B.BOM_F32))


def test_sharded_step_calls_refuse_a_null_handle(built):
    """The row- and vocabulary-sharded parts check the handle before anything
    else (no device is touched)."""
    P = [ALIGNED]
    assert _code(B.bom_step_shard_begin, None, ALIGNED, ALIGNED, 4, P, ALIGNED, stream=0) == B.BOM_EINVAL
    assert _code(B.bom_step_vshard_begin, None, ALIGNED, ALIGNED, 4, P, 10, 0, ALIGNED, stream=0) == B.BOM_EINVAL
    assert _code(B.bom_step_vshard_mid, None, ALIGNED, ALIGNED, 4, P, ALIGNED, 1, ALIGNED, 2, [ALIGNED], ALIGNED,
                 stream=0) == B.BOM_EINVAL
    assert _code(B.bom_step_vshard_end, None, ALIGNED, ALIGNED, 4, P, ALIGNED, [ALIGNED], stream=0) == B.BOM_EINVAL
