"""C ABI checks that need no GPU: the library builds, loads, exports every declared symbol, and
validates arguments on the host before touching a device."""
import ctypes as C
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2512_14681_gb300 import build as B
    from paper_2512_14681_gb300 import _lib

    B.build()
    return _lib.load()


def declared_symbols():
    names = set()
    for f in os.listdir(os.path.join(ROOT, "include")):
        if not f.endswith(".h"):
            continue
        text = open(os.path.join(ROOT, "include", f)).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        for m in re.finditer(r"^\s*(?:jf_status|void|const char\*)\s+(jf_\w+)\s*\(", text, flags=re.M):
            names.add(m.group(1))
    return names


def test_every_declared_symbol_is_exported(lib):
    from paper_2512_14681_gb300 import _lib

    names = declared_symbols()
    assert len(names) >= 19
    assert names == set(_lib.EXPORTS)
    for n in names:
        assert getattr(lib, n) is not None


def _cfg(shape):
    from paper_2512_14681_gb300 import jacobi as JJ

    return JJ.model_config(shape)


def test_arena_bytes_host_only(lib):
    from paper_2512_14681_gb300 import _lib as J
    from paper_2512_14681_gb300 import inputs as I

    out = C.c_size_t()
    rc = J.RuntimeConfig(1, 2048, 64, 0, None, 0, None)
    assert lib.jf_arena_bytes(C.byref(_cfg(I.QWEN7B_BF16)), C.byref(rc), C.byref(out)) == J.JF_OK
    assert out.value > I.QWEN7B_BF16.weight_bytes() + 2 * 28 * 4 * 128 * 2 * 2048
    assert out.value < I.QWEN7B_BF16.weight_bytes() * 1.2
    rc2 = J.RuntimeConfig(1, 256, 32, 32, None, 0, None)
    assert lib.jf_arena_bytes(C.byref(_cfg(I.TINY_F32)), C.byref(rc2), C.byref(out)) == J.JF_OK
    assert out.value > I.TINY_F32.weight_bytes()


def test_invalid_configs_rejected_on_host(lib):
    from paper_2512_14681_gb300 import _lib as J
    from paper_2512_14681_gb300 import inputs as I

    out = C.c_size_t()
    rc = J.RuntimeConfig(1, 2048, 64, 0, None, 0, None)
    bad = _cfg(I.QWEN7B_BF16)
    bad.head_dim = 64
    assert lib.jf_arena_bytes(C.byref(bad), C.byref(rc), C.byref(out)) == J.JF_EUNSUPPORTED
    bad = _cfg(I.QWEN7B_BF16)
    bad.n_kv_heads = 5
    assert lib.jf_arena_bytes(C.byref(bad), C.byref(rc), C.byref(out)) == J.JF_EUNSUPPORTED
    bad = _cfg(I.QWEN7B_BF16)
    bad.dtype = 7
    assert lib.jf_arena_bytes(C.byref(bad), C.byref(rc), C.byref(out)) == J.JF_EINVAL
    for field in ("qkv_bias", "tie_embeddings"):
        bad = _cfg(I.QWEN7B_BF16)
        setattr(bad, field, 2)
        assert lib.jf_arena_bytes(C.byref(bad), C.byref(rc), C.byref(out)) == J.JF_EINVAL, field
    # a tied LM head needs no arena of its own: exactly one [V, d] matrix less
    untied, tied = _cfg(I.QWEN7B_BF16), _cfg(I.QWEN7B_BF16)
    untied.tie_embeddings, tied.tie_embeddings = 0, 1
    a_u, a_t = C.c_size_t(), C.c_size_t()
    assert lib.jf_arena_bytes(C.byref(untied), C.byref(rc), C.byref(a_u)) == J.JF_OK
    assert lib.jf_arena_bytes(C.byref(tied), C.byref(rc), C.byref(a_t)) == J.JF_OK
    assert 0 <= a_u.value - a_t.value - 152064 * 3584 * 2 < 4096
    rc_bad = J.RuntimeConfig(0, 2048, 64, 0, None, 0, None)
    assert lib.jf_arena_bytes(C.byref(_cfg(I.QWEN7B_BF16)), C.byref(rc_bad), C.byref(out)) == J.JF_EINVAL
    for page_size, want in ((16, J.JF_OK), (0, J.JF_OK), (32, J.JF_EUNSUPPORTED), (8, J.JF_EUNSUPPORTED)):
        r = J.RuntimeConfig(1, 2048, 64, 0, None, 0, None, page_size)
        assert lib.jf_arena_bytes(C.byref(_cfg(I.QWEN7B_BF16)), C.byref(r), C.byref(out)) == want, page_size
    for max_segments, want in ((0, J.JF_OK), (1, J.JF_OK), (256, J.JF_OK), (257, J.JF_EINVAL), (-1, J.JF_EINVAL)):
        r = J.RuntimeConfig(1, 2048, 64, 0, None, 0, None, 16, max_segments)
        assert lib.jf_arena_bytes(C.byref(_cfg(I.QWEN7B_BF16)), C.byref(r), C.byref(out)) == want, max_segments
    # max_segments sizes the attention's lane-state scratch: more segments, a larger arena
    small, large = C.c_size_t(), C.c_size_t()
    lib.jf_arena_bytes(C.byref(_cfg(I.QWEN7B_BF16)), C.byref(J.RuntimeConfig(1, 2048, 64, 0, None, 0, None, 16, 2)),
                       C.byref(small))
    lib.jf_arena_bytes(C.byref(_cfg(I.QWEN7B_BF16)), C.byref(J.RuntimeConfig(1, 2048, 64, 0, None, 0, None, 16, 64)),
                       C.byref(large))
    assert large.value > small.value
    rc_bad = J.RuntimeConfig(1, 2048, 64, 65, None, 0, None)
    assert lib.jf_arena_bytes(C.byref(_cfg(I.QWEN7B_BF16)), C.byref(rc_bad), C.byref(out)) == J.JF_EINVAL
    # a context needs an arena
    h = C.c_void_p()
    assert lib.jf_create(C.byref(_cfg(I.TINY_F32)), C.byref(rc), C.byref(h)) == J.JF_ENOMEM
    assert not h.value


def test_op_gemm_validation_and_workspace(lib):
    from paper_2512_14681_gb300 import _lib as J

    nb = C.c_size_t()
    assert lib.jf_op_gemm_workspace_bytes(3584, 3584, 32, 0, C.byref(nb)) == J.JF_OK
    assert nb.value >= 28 * 5 * 32 * 128 * 4
    assert lib.jf_op_gemm_workspace_bytes(0, 3584, 32, 0, C.byref(nb)) == J.JF_EINVAL
    # K not a multiple of 8 (16-byte TMA rows) and null pointers are refused before any launch
    assert lib.jf_op_gemm(J.JF_BF16, 16, 16, 16, 128, 60, 4, 0, 16, 1 << 20, 16, None) == J.JF_EINVAL
    assert lib.jf_op_gemm(J.JF_BF16, None, 16, 16, 128, 64, 4, 0, 16, 1 << 20, 16, None) == J.JF_EINVAL


def test_null_context_is_refused_without_touching_a_device(lib):
    """Every call that takes a context refuses a null one with JF_EINVAL (host check, no CUDA call)."""
    from paper_2512_14681_gb300 import _lib as J

    one = (C.c_int32 * 4)(1, 2, 3, 4)
    out = (C.c_int32 * 4)()
    f = (C.c_float * 4)()
    n = C.c_int()
    d = C.c_double()
    ll = C.c_longlong()
    blk = J.Block(0, 0, 1, -1)
    gp = J.GenParams()
    calls = {
        "jf_init_random_weights": (None, 0, 0.02),
        "jf_load_weights": (None, b"/nonexistent"),
        "jf_save_weights": (None, b"/nonexistent"),
        "jf_get_weights": (None, 0, 0, 1, f),
        "jf_prefill": (None, 0, one, 4, out),
        "jf_truncate": (None, 0, 0),
        "jf_seq_len": (None, 0, C.byref(n)),
        "jf_jacobi_step": (None, 0, 1, C.byref(blk), one, out, out, out, None, None),
        "jf_forward_logits": (None, 0, 1, one, None, None, out),
        "jf_generate": (None, 1, None, one, C.byref(gp), out, None),
        "jf_generate_device": (None, 1, None, one, C.byref(gp), None, None),
        "jf_set_profiling": (None, 1),
        "jf_kernel_time": (None, 0, C.byref(d), C.byref(ll)),
        "jf_set_wait_limit": (None, 2_000_000_000),
        "jf_wait_limit_probe": (None, None),
    }
    for name, args in calls.items():
        assert getattr(lib, name)(*args) == J.JF_EINVAL, name
    assert lib.jf_last_error(None) == b"null context"
    lib.jf_destroy(None)
