"""The C-ABI library loads and exports every entry point include/starkv.h
declares; host-side checks that need no GPU.  CPU only."""
import ctypes
import re
from pathlib import Path

import pytest

from paper_2606_01790_gb300 import build as B
from paper_2606_01790_gb300 import starkv as sk

ROOT = Path(__file__).resolve().parents[1]


@pytest.fixture(scope="module")
def library():
    B.build()
    return sk.lib()


def declared_functions():
    text = (ROOT / "include" / "starkv.h").read_text()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(starkv_[a-z_]+)\s*\(", text)))


def test_header_declares_the_expected_calls():
    names = declared_functions()
    for required in ("starkv_init_state", "starkv_score_layer", "starkv_select", "starkv_compact",
                     "starkv_step"):
        assert required in names
    assert set(names) == set(sk.ABI_FUNCTIONS)


def test_library_exports_every_declared_symbol(library):
    for name in declared_functions():
        assert hasattr(library, name), name
        assert ctypes.cast(getattr(library, name), ctypes.c_void_p).value


def test_struct_layouts_match_header():
    assert ctypes.sizeof(sk.CConfig) == 13 * 4 + 10 * 4 + 4 * 4
    assert [f[0] for f in sk.CConfig._fields_][-4:] == ["select_mode", "decay_mode", "aeb_mode", "mi_span"]


def test_header_constants_match_binding():
    import re
    text = (ROOT / "include" / "starkv.h").read_text()
    m = re.search(r"#define STARKV_STATS_STRIDE\(G\) \(8 \+ (\d+) \* \(G\)\)", text)
    assert m and all(sk.stats_stride(g) == 8 + int(m.group(1)) * g for g in range(1, 9))
    m = re.search(r"STARKV_SELECT_GLOBAL = (\d+), STARKV_SELECT_PER_HEAD = (\d+)", text)
    assert m and (int(m.group(1)), int(m.group(2))) == (sk.SELECT_GLOBAL, sk.SELECT_PER_HEAD)
    assert ctypes.sizeof(sk.CSeq) == 4 * 8 + 8 + 4 * 4 + 7 * 8 + 8 + 8 + 2 * 8


def test_default_config_matches_paper_defaults(library):
    c = sk.Config.default()
    assert (c.n_heads, c.n_kv_heads, c.head_dim, c.window) == (28, 4, 128, 32)
    assert abs(c.lambda_ - 0.5) < 1e-7 and abs(c.delta - 0.2) < 1e-7 and abs(c.d_min - 0.1) < 1e-7
    assert (c.n_warmup, c.n_ramp) == (5, 10)
    assert abs(c.t_min - 0.95) < 1e-7 and abs(c.t_max - 1.05) < 1e-7
    assert c.select_mode == sk.SELECT_GLOBAL


@pytest.mark.parametrize("bad", [dict(head_dim=64), dict(n_heads=30), dict(window=64),
                                 dict(pool_kernel=4), dict(mi_bins=1), dict(t_min=0.0),
                                 dict(n_kv_heads=0), dict(grid_rows=2000), dict(select_mode=2),
                                 dict(decay_mode=3), dict(aeb_mode=2), dict(mi_span=-1),
                                 dict(n_heads=40, n_kv_heads=40, window=4),
                                 dict(n_kv_heads=28, select_mode=1)])
def test_invalid_config_rejected_before_any_device_call(library, bad):
    cfg = sk.Config(**bad)
    with pytest.raises(sk.StarkvError) as e:
        sk.State(cfg, stream=0)
    assert e.value.status in (sk.ERR_INVALID_ARG, sk.ERR_UNSUPPORTED)


def test_meta_packing_roundtrip():
    import numpy as np
    vis = np.array([0, 1, 1, 1]); fr = np.array([0, 3, 2047, 0])
    row = np.array([0, 51, 1023, 7]); col = np.array([0, 0, 9, 1023])
    w = sk.pack_meta(vis, fr, row, col)
    assert w[0] == 0 and (w[1:] >> 31).tolist() == [1, 1, 1]
    v2, f2, r2, c2 = sk.unpack_meta(w)
    assert v2.tolist() == vis.tolist() and f2[1:].tolist() == fr[1:].tolist()
    assert r2[1:].tolist() == row[1:].tolist() and c2[1:].tolist() == col[1:].tolist()
    with pytest.raises(ValueError):
        sk.pack_meta([1], [4096], [0], [0])


def test_wait_selftest_checks_its_arguments_on_the_host(library):
    assert library.starkv_selftest_wait(None, 1000000, None) == sk.ERR_INVALID_ARG


def test_header_compiles_as_c_and_its_layouts_match_the_binding(tmp_path):
    """The header alone, compiled by the host C compiler: struct sizes, the
    slot-state size macro and the constants, against the ctypes mirror."""
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    src = tmp_path / "probe.c"
    src.write_text(
        '#include <stdio.h>\n#include "starkv.h"\n'
        "int main(void) {\n"
        '  printf("%zu %zu %zu %zu %u %d\\n", sizeof(starkv_config), sizeof(starkv_seq),\n'
        "         sizeof(starkv_slot_header), (size_t)STARKV_SLOT_STATE_BYTES(28, 4, 2704),\n"
        "         (unsigned)STARKV_SLOT_MAGIC, (int)STARKV_STATS_STRIDE(4));\n"
        "  return 0;\n}\n")
    exe = tmp_path / "probe"
    subprocess.run([cc, "-std=c99", "-Wall", "-Werror", f"-I{ROOT / 'include'}", str(src), "-o", str(exe)],
                   check=True, capture_output=True)
    got = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.split()
    want = [ctypes.sizeof(sk.CConfig), ctypes.sizeof(sk.CSeq), ctypes.sizeof(sk.CSlotHeader),
            sk.slot_state_bytes_for(28, 4, 2704), sk.SLOT_MAGIC, sk.stats_stride(4)]
    assert [int(x) for x in got] == want


def test_slot_calls_check_their_arguments_on_the_host(library):
    n = ctypes.c_size_t(0)
    assert library.starkv_slot_state_bytes(None, ctypes.byref(n)) == sk.ERR_INVALID_ARG
    buf = (ctypes.c_uint8 * 64)()
    assert library.starkv_export_slot(None, 0, buf, 64, None) == sk.ERR_INVALID_ARG
    assert library.starkv_import_slot(None, 0, buf, 64, None) == sk.ERR_INVALID_ARG
