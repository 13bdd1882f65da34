"""The C-ABI library builds, loads, exports every declared symbol, and rejects
bad arguments on the host (no GPU needed for any of this)."""
import ctypes
import glob
import os
import re
import shutil

import pytest

from paper_2609_01068_gb300 import build as B
from paper_2609_01068_gb300 import outlets as O

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared_functions():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        text = open(h).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        for m in re.finditer(r"^\s*[A-Za-z_][\w\s\*]*?\b(outlets_\w+)\s*\(", text, flags=re.M):
            names.add(m.group(1))
    return sorted(names)


@pytest.fixture(scope="module")
def built_lib():
    if not os.path.exists(B.LIB_PATH) and not shutil.which("nvcc") and not os.path.exists("/usr/local/cuda/bin/nvcc"):
        pytest.skip("nvcc unavailable and library not built")
    B.build()
    return O.load()


def test_header_declares_the_entry_points():
    names = _declared_functions()
    for must in ("outlets_create", "outlets_predict_prefill", "outlets_predict_step", "outlets_kv_create",
                 "outlets_destroy", "outlets_last_error", "outlets_predict_prefill_dual",
                 "outlets_predict_step_dual", "outlets_draft_head", "outlets_predict_prefill_ex",
                 "outlets_predict_step_ex", "outlets_predict_draft_step", "outlets_kv_truncate"):
        assert must in names


def test_library_exports_every_declared_symbol(built_lib):
    for name in _declared_functions():
        assert hasattr(built_lib, name), name


def test_create_rejects_invalid_config_on_host(built_lib):
    cfg = O.Config()
    cfg.d_model, cfg.n_heads, cfg.n_kv_heads, cfg.head_dim, cfg.ffn_dim = 100, 4, 2, 64, 688  # d not % 64
    cfg.n_head_hidden = 1
    cfg.head_hidden[0] = 128
    cfg.rope_theta, cfg.rms_eps, cfg.dtype = 1e4, 1e-5, O.F32
    cfg.max_tokens, cfg.max_batch, cfg.max_position = 16, 4, 64
    w = O.Weights()
    h = ctypes.c_void_p()
    assert built_lib.outlets_create(ctypes.byref(cfg), ctypes.byref(w), ctypes.byref(h)) == O.EINVAL
    assert not h.value
    cfg.d_model = 256
    cfg.n_kv_heads = 3  # H % KVH != 0
    assert built_lib.outlets_create(ctypes.byref(cfg), ctypes.byref(w), ctypes.byref(h)) == O.EINVAL
    cfg.n_kv_heads = 2
    cfg.dtype = O.BF16
    cfg.head_dim = 96  # bf16 attention supports 64 / 128
    assert built_lib.outlets_create(ctypes.byref(cfg), ctypes.byref(w), ctypes.byref(h)) == O.EINVAL
    cfg.head_dim = 64
    # every weight pointer set (never read: the config is checked first), so
    # only the draft head width makes these configurations invalid
    dummy = (ctypes.c_float * 4)()
    for name, _ in O.Weights._fields_:
        if name in ("head_w", "head_b"):
            for i in range(cfg.n_head_hidden + 1):
                getattr(w, name)[i] = ctypes.addressof(dummy)
        else:
            setattr(w, name, ctypes.addressof(dummy))
    for vocab in (5, -1, 262145):  # outside 8 .. 262144
        cfg.vocab = vocab
        assert built_lib.outlets_create(ctypes.byref(cfg), ctypes.byref(w), ctypes.byref(h)) == O.EINVAL
        assert not h.value
    cfg.vocab = 0
    cfg.embed_vocab = -3
    assert built_lib.outlets_create(ctypes.byref(cfg), ctypes.byref(w), ctypes.byref(h)) == O.EINVAL
    assert not h.value


def test_null_handles_are_rejected(built_lib):
    z = (ctypes.c_float * 4)()
    cu = (ctypes.c_int32 * 2)(0, 4)
    taps = (ctypes.c_void_p * 3)()
    assert built_lib.outlets_predict_prefill(None, taps, cu, 1, 4, None, None, 0, z, None, None) == O.EINVAL
    assert built_lib.outlets_predict_step(None, taps, 1, None, None, z, None, None) == O.EINVAL
    d = O.DraftOut()
    assert built_lib.outlets_predict_prefill_dual(None, taps, cu, 1, 4, None, None, 0, z, None, ctypes.byref(d),
                                                  None) == O.EINVAL
    assert built_lib.outlets_predict_step_dual(None, taps, 1, None, None, z, None, ctypes.byref(d), None) == O.EINVAL
    assert built_lib.outlets_draft_head(None, None, 1, ctypes.byref(d), None) == O.EINVAL
    assert built_lib.outlets_predict_prefill_ex(None, taps, None, cu, 1, 4, None, None, 0, z, None, None,
                                                None) == O.EINVAL
    assert built_lib.outlets_predict_step_ex(None, taps, None, 1, None, None, z, None, None, None) == O.EINVAL
    assert built_lib.outlets_predict_draft_step(None, None, 1, None, None, z, None, None, None) == O.EINVAL
    assert built_lib.outlets_kv_truncate(None, 0, 0) == O.EINVAL
    assert built_lib.outlets_kv_reset_slot(None, 0) == O.EINVAL
    assert built_lib.outlets_kv_slot_length(None, 0) == -1
    assert built_lib.outlets_kv_free_pages(None) == -1
    assert built_lib.outlets_check(None, None) == O.EINVAL
    info = O.TensorInfo()
    assert built_lib.outlets_get_intermediate(None, 0, None, 0, ctypes.byref(info), None) == O.EINVAL
