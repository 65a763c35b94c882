"""The C ABI on a machine without a GPU: libqk.so builds, loads, exports every
function include/*.h declares, and its host-only entry points (presets, tensor
counts, packed sizes, argument validation, error strings) behave as declared.
No call here touches a device."""
import ctypes
import glob
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2609_12471_gb300 import build
    path = build.build()
    return ctypes.CDLL(path)


def _declared():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        src = open(h).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        names |= set(re.findall(r"^\s*(?:const\s+)?[\w]+\s*\**\s+\**(qk_\w+)\s*\(", src, flags=re.M))
    return names


def test_every_declared_symbol_is_exported(lib):
    names = _declared()
    assert len(names) >= 18, names
    missing = [n for n in sorted(names) if not hasattr(lib, n)]
    assert not missing, f"declared but not exported: {missing}"


def test_binding_covers_the_declared_abi():
    import paper_2609_12471_gb300 as qk
    assert set(qk.exported_symbols()) == _declared()


def test_presets_and_sizes():
    import paper_2609_12471_gb300 as qk
    c = qk.qk_config_preset("q8b")
    assert (c.n_layers, c.hidden, c.n_q_heads, c.n_kv_heads, c.head_dim, c.intermediate,
            c.vocab, c.dtype) == (36, 4096, 32, 8, 128, 12288, 151936, qk.QK_DTYPE_BF16)
    assert c.rms_eps == 1e-6 and c.rope_theta == 1e6
    assert qk.qk_weight_count(c) == 3 + 11 * 36
    # bf16 weights (8.19e9 params) + fp32 gains + RoPE tables + alignment
    nbytes = qk.qk_model_packed_bytes(c)
    params = 2 * 151936 * 4096 + 36 * (192937984) 
    assert 2 * params < nbytes < 2 * params + 64 * 2**20
    t = qk.qk_config_preset("tiny_fp32")
    assert (t.n_layers, t.hidden, t.dtype) == (2, 256, qk.QK_DTYPE_F32)
    one = qk.qk_config_preset("q8b_layer")
    assert one.n_layers == 1 and qk.qk_weight_count(one) == 14


@pytest.mark.parametrize("field,value,code", [
    ("dtype", 7, -3), ("head_dim", 96, -3), ("hidden", 100, -2), ("intermediate", 100, -2),
    ("vocab", 3, -2), ("n_kv_heads", 3, -2), ("reserved", 1, -1), ("max_positions", 0, -1),
])
def test_config_validation_errors(field, value, code):
    import paper_2609_12471_gb300 as qk
    c = qk.qk_config_preset("q8b")
    setattr(c, field, value)
    with pytest.raises(qk.QKError) as e:
        qk.qk_model_packed_bytes(c)
    assert e.value.code == code
    assert qk.qk_last_error()


def test_unknown_preset_and_null_arguments(lib):
    import paper_2609_12471_gb300 as qk
    with pytest.raises(qk.QKError) as e:
        qk.qk_config_preset("nope")
    assert e.value.code == qk.QK_EINVAL and "nope" in str(e.value)
    lib.qk_model_packed_bytes.argtypes = [ctypes.c_void_p, ctypes.c_void_p]
    assert lib.qk_model_packed_bytes(None, None) == qk.QK_EINVAL
    lib.qk_workspace_bytes.argtypes = [ctypes.c_void_p] + [ctypes.c_int] * 4 + [ctypes.c_void_p]
    assert lib.qk_workspace_bytes(None, 0, 1, 1, 1, None) == qk.QK_EINVAL


def test_grpo_and_turn_entry_points_validate_on_the_host(lib):
    """Argument errors of the GRPO, sampling and multi-turn entry points come back
    before any device work (fake non-null pointers are never dereferenced)."""
    import paper_2609_12471_gb300 as qk
    assert qk.qk_grpo_workspace_bytes(1) == 256
    assert qk.qk_grpo_workspace_bytes(1000) == 8192
    with pytest.raises(qk.QKError) as e:
        qk.qk_grpo_workspace_bytes(0)
    assert e.value.code == qk.QK_ESHAPE
    P = 16  # a fake, aligned, never-dereferenced device address
    args = dict(lp=P, lp_old=P, lp_ref=P, B=6, T=4, ld=4, rewards=P, group=3, mask=None,
                eps_low=0.2, eps_high=0.28, beta=0.01, loss_tok=P)

    def call(**over):
        a = dict(args, **over)
        with pytest.raises(qk.QKError) as e:
            qk.qk_grpo_token_loss(a["lp"], a["lp_old"], a["lp_ref"], a["B"], a["T"], a["ld"],
                                  a["rewards"], a["group"], a["mask"], a["eps_low"], a["eps_high"],
                                  a["beta"], a["loss_tok"], None, None, 0, stream=0)
        return e.value.code

    assert call(lp=None) == qk.QK_EINVAL
    assert call(lp_ref=None) == qk.QK_EINVAL          # beta != 0 needs a reference policy
    assert call(group=4) == qk.QK_ESHAPE              # 6 rows are not whole groups of 4
    assert call(ld=3) == qk.QK_ESHAPE                 # row stride below T
    assert call(eps_low=1.5) == qk.QK_EINVAL
    assert call() == qk.QK_ENOSPACE                   # valid arguments, no workspace
    with pytest.raises(qk.QKError) as e:
        qk.qk_rollout_sampled(None, P, 1, 8, P, 1, 4, 2, 1.0, 0, P, P, ws_bytes=0, stream=0)
    assert e.value.code == qk.QK_EINVAL
    with pytest.raises(qk.QKError) as e:
        qk.qk_prefill_rows(None, P, 1, 8, P, 1, 4, P, ws_bytes=0, stream=0)
    assert e.value.code == qk.QK_EINVAL


def test_backward_entry_points_validate_on_the_host(lib):
    """qk_grpo_coef and qk_backward_logprob reject bad arguments before any device work."""
    import paper_2609_12471_gb300 as qk
    P = 16
    with pytest.raises(qk.QKError) as e:
        qk.qk_grpo_coef(None, P, P, 6, 4, 4, P, 3, None, 0.2, 0.28, 0.01, P, P, None, None, 0, stream=0)
    assert e.value.code == qk.QK_EINVAL
    with pytest.raises(qk.QKError) as e:  # 6 rows are not whole groups of 4
        qk.qk_grpo_coef(P, P, P, 6, 4, 4, P, 4, None, 0.2, 0.28, 0.01, P, P, None, None, 0, stream=0)
    assert e.value.code == qk.QK_ESHAPE
    with pytest.raises(qk.QKError) as e:  # valid arguments, no workspace
        qk.qk_grpo_coef(P, P, P, 6, 4, 4, P, 3, None, 0.2, 0.28, 0.01, P, P, None, None, 0, stream=0)
    assert e.value.code == qk.QK_ENOSPACE
    with pytest.raises(qk.QKError) as e:
        qk.qk_backward_logprob(None, P, 1, 4, P, [P] * 25, ws_bytes=0, stream=0)
    assert e.value.code == qk.QK_EINVAL
    assert qk.QK_CALL_BACKWARD == 4


def test_debug_hook_validates_on_the_host():
    import paper_2609_12471_gb300 as qk
    with pytest.raises(qk.QKError) as e:
        qk.qk_debug_expire_next_wait(None, 1000)
    assert e.value.code == qk.QK_EINVAL


def test_paged_entry_points_validate_on_the_host(lib):
    """The paged-cache calls reject a missing model or pages before any device work, and
    the binding's qk_kv_pages has the header's layout (pointer, three int32)."""
    import paper_2609_12471_gb300 as qk
    assert ctypes.sizeof(qk.qk_kv_pages) == 24
    assert [f for f, _ in qk.qk_kv_pages._fields_] == ["table", "per_row", "n_pages", "page_size"]
    P = 256
    for call in (lambda: qk.qk_kv_pages_bytes(None, 4, 128),
                 lambda: qk.qk_decode_step_paged(None, P, P, 2, 4, 128, P, P, 2, ws_bytes=0, stream=0),
                 lambda: qk.qk_prefill_rows_paged(None, P, P, 2, 4, 128, P, 2, 8, P, ws_bytes=0, stream=0)):
        with pytest.raises(qk.QKError) as e:
            call()
        assert e.value.code == qk.QK_EINVAL
    assert qk.QK_STATUS_BAD_PAGE == 8
