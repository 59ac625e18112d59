"""The C-ABI library builds, loads without a GPU, exports every symbol the
header declares, and its host-only logic behaves as documented."""
import ctypes
import json
import os
import re
import subprocess
import tempfile

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "buddy.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2606_09514_gb300 import build as b
    b.build()
    import paper_2606_09514_gb300 as pkg
    return pkg.load_library()


def _declared():
    txt = open(HEADER).read()
    return sorted(set(re.findall(r"BUDDY_API\s+[\w\s\*]+?\b(buddy_\w+)\s*\(", txt)))


def test_every_declared_symbol_is_exported(lib):
    names = _declared()
    assert len(names) >= 10
    for n in names:
        assert hasattr(lib, n), n
    from paper_2606_09514_gb300 import binding
    assert sorted(binding.EXPORTED) == names


def test_budget_to_k_matches_paper_settings(lib):
    with open(os.path.join(ROOT, "tests", "golden", "budget_k.json")) as f:
        g = json.load(f)
    from oracle import buddy_oracle as O
    for c in g["cases"]:
        assert lib.buddy_budget_to_k(c["b"], c["L"]) == c["k"]
    for L in (3, 8, 28, 32, 40):
        for b in [i / 64 for i in range(0, 70)]:
            assert lib.buddy_budget_to_k(b, L) == O.budget_to_k(b, L), (b, L)
    assert lib.buddy_budget_to_k(0.5, 2) == -1
    assert lib.buddy_budget_to_k(float("nan"), 32) == -1


def test_invalid_configs_rejected_before_any_cuda_call(lib):
    from paper_2606_09514_gb300 import binding as B
    h = ctypes.c_void_p()
    assert lib.buddy_create(None, ctypes.byref(h)) == B.BUDDY_ERR_ARG
    good = dict(n_layers=8, d_model=256, n_q_heads=4, n_kv_heads=4, head_dim=64, ffn_dim=704, dm_hidden=16,
                dtype=0, max_batch=4, max_pos=64, qkv_bias=0, rms_eps=1e-5, rope_theta=1e4)
    bad_cases = [dict(n_layers=2), dict(head_dim=96), dict(n_kv_heads=3), dict(d_model=320),
                 dict(ffn_dim=700), dict(ffn_dim=0), dict(max_batch=0), dict(max_batch=5000), dict(max_pos=0),
                 dict(dtype=7), dict(rms_eps=0.0), dict(n_q_heads=36, n_kv_heads=4, d_model=36 * 64),
                 dict(feature=3), dict(feature=-1), dict(ctx_layer=6), dict(ctx_layer=-1), dict(skip_kv=2),
                 dict(max_prefill_tokens=-1), dict(max_prefill_tokens=70000), dict(dtype=1, max_batch=257)]
    for bad in bad_cases:
        cfg = B.buddy_config(**{**good, **bad})
        assert lib.buddy_create(ctypes.byref(cfg), ctypes.byref(h)) == B.BUDDY_ERR_ARG, bad
    assert lib.buddy_set_weights(None, None, None) == B.BUDDY_ERR_ARG
    assert lib.buddy_decode_step(None, None, 1, None, None, None, None, None, None, None, None) == B.BUDDY_ERR_ARG
    assert lib.buddy_route(None, None, 1, None, None, None, None, None, None) == B.BUDDY_ERR_ARG
    assert lib.buddy_kv_append(None, None, 0, 1, None, 1, None, None, 0, None) == B.BUDDY_ERR_ARG
    assert lib.buddy_set_budget_predictor(None, None) == B.BUDDY_ERR_ARG
    assert lib.buddy_error_string(B.BUDDY_ERR_RANGE) == b"value out of range"
    assert lib.buddy_version() >= 1


def test_ctypes_structs_match_c_layout():
    """sizeof/offsetof of the header's structs (compiled with gcc) equal the
    binding's ctypes layouts."""
    from paper_2606_09514_gb300 import binding as B
    structs = {"buddy_config": B.buddy_config, "buddy_layer_weights": B.buddy_layer_weights,
               "buddy_dm_weights": B.buddy_dm_weights, "buddy_kv_state": B.buddy_kv_state,
               "buddy_predictor_weights": B.buddy_predictor_weights}
    lines = ['#include <stdio.h>', '#include <stddef.h>', f'#include "{HEADER}"', 'int main(void){']
    for n, cls in structs.items():
        lines.append(f'printf("{n} %zu\\n", sizeof({n}));')
        for f, _ in cls._fields_:
            lines.append(f'printf("{n}.{f} %zu\\n", offsetof({n}, {f}));')
    lines.append("return 0;}")
    with tempfile.TemporaryDirectory() as d:
        src = os.path.join(d, "l.c")
        exe = os.path.join(d, "l")
        open(src, "w").write("\n".join(lines))
        subprocess.run(["gcc", "-o", exe, src], check=True)
        out = subprocess.run([exe], capture_output=True, text=True, check=True).stdout.split("\n")
    got = dict(l.split() for l in out if l)
    for n, cls in structs.items():
        assert int(got[n]) == ctypes.sizeof(cls), n
        for f, _ in cls._fields_:
            assert int(got[f"{n}.{f}"]) == getattr(cls, f).offset, (n, f)


def test_profiler_class_names_match_binding(lib):
    """The binding's names for the profiler's kernel classes are the library's,
    in the order of the header's enum."""
    from paper_2606_09514_gb300 import binding
    txt = open(HEADER).read()
    enum = re.search(r"enum\s*\{\s*(BUDDY_PROF_CHECK[^}]*)\}", txt).group(1)
    n_cls = len(re.findall(r"\bBUDDY_PROF_(?!NCLASS)\w+", enum))
    assert n_cls == len(binding.PROF_CLASSES)
    lib.buddy_profile_class_name.restype = ctypes.c_char_p
    lib.buddy_profile_class_name.argtypes = [ctypes.c_int32]
    names = [lib.buddy_profile_class_name(i).decode() for i in range(n_cls)]
    assert names == binding.PROF_CLASSES
    assert lib.buddy_profile_class_name(n_cls).decode() == "unknown"
