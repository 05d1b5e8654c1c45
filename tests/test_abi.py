"""The C ABI library loads, exports every symbol include/ntc.h declares, and
rejects bad arguments on the host (no GPU needed for any of this)."""
import ctypes
import os
import re

import pytest

from paper_2608_27888_gb300 import build as B

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    path = B.build()
    return ctypes.CDLL(path)


def declared():
    src = open(os.path.join(ROOT, "include", "ntc.h")).read()
    return re.findall(r"NTC_API\s+[\w\s\*]+?\b(ntc_\w+)\s*\(", src)


def test_every_declared_symbol_is_exported(lib):
    names = declared()
    assert len(names) >= 13
    for n in names:
        assert hasattr(lib, n), n


def test_binding_mirrors_the_abi():
    from paper_2608_27888_gb300 import ntc
    names = declared()
    assert sorted(ntc.EXPORTS) == sorted(names)
    for n in names:
        if n not in ("ntc_status_string",):
            assert hasattr(ntc, n), n


def test_host_side_validation(lib):
    lib.ntc_create.argtypes = [ctypes.c_void_p, ctypes.c_void_p]
    lib.ntc_last_error.restype = ctypes.c_char_p
    ctx = ctypes.c_void_p(123)
    assert lib.ntc_create(None, ctypes.byref(ctx)) == 1
    assert ctx.value is None
    assert b"null descriptor" in lib.ntc_last_error()
    from paper_2608_27888_gb300 import ntc
    d = ntc.ntc_desc()
    assert lib.ntc_create(ctypes.byref(d), ctypes.byref(ctx)) == 1  # null arrays
    lib.ntc_decode.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p,
                               ctypes.c_void_p, ctypes.c_int]
    assert lib.ntc_decode(None, None, 0, None, None, 0) == 1
    lib.ntc_destroy.argtypes = [ctypes.c_void_p]
    assert lib.ntc_destroy(None) == 0
    lib.ntc_max_tiles.restype = ctypes.c_size_t
    lib.ntc_max_tiles.argtypes = [ctypes.c_void_p, ctypes.c_size_t]
    assert lib.ntc_max_tiles(None, 1000) == 0
    lib.ntc_status_string.restype = ctypes.c_char_p
    assert lib.ntc_status_string(2) == b"unsupported"


def test_descriptor_validation_before_any_device_work(lib):
    import numpy as np
    from paper_2608_27888_gb300 import ntc
    from tests.util import tiny_assets
    a = tiny_assets([[(8, 8), (4, 4)]], hidden=64, out_dim=8)
    keep = [np.ascontiguousarray(x) for x in (a.level_dims, a.latent_offsets, a.latents, a.weights,
                                              a.set_to_decoder)]

    def desc(**over):
        d = ntc.ntc_desc(num_sets=1, num_decoders=1, latent_channels=8, num_levels=2, num_mips=1,
                         level_dims=keep[0].ctypes.data, latent_offsets=keep[1].ctypes.data,
                         latents=keep[2].ctypes.data, num_texels=keep[2].size // 8, in_dim=16,
                         hidden=64, num_hidden_layers=2, out_dim=8, weights=keep[3].ctypes.data,
                         set_to_decoder=keep[4].ctypes.data, precision=0, address_mode=0)
        for k, v in over.items():
            setattr(d, k, v)
        return d
    ctx = ctypes.c_void_p()
    for bad, status in [(dict(hidden=96), 2), (dict(latent_channels=6), 2), (dict(num_levels=3), 2),
                        (dict(out_dim=17), 2), (dict(num_decoders=0), 1), (dict(num_mips=0), 1),
                        (dict(num_texels=10), 1), (dict(address_mode=2), 1), (dict(precision=9), 1),
                        (dict(num_hidden_layers=5), 2), (dict(num_hidden_layers=0), 2),
                        (dict(latent_channels=4), 1),          # in_dim no longer levels x channels
                        (dict(pe_frequencies=2), 1),           # in_dim misses the 8 encoding inputs
                        (dict(pe_frequencies=9, in_dim=52), 2), (dict(activation=2), 1),
                        (dict(activation=1, leaky_slope=float("inf")), 1),
                        (dict(output_format=2), 1),            # neither fp32 nor fp16 rows
                        (dict(output_format=1, precision=2), 2)]:  # fp16 rows need a tensor-core precision
        assert lib.ntc_create(ctypes.byref(desc(**bad)), ctypes.byref(ctx)) == status, bad
    keep[4][0] = 1  # map entry beyond num_decoders
    assert lib.ntc_create(ctypes.byref(desc()), ctypes.byref(ctx)) == 1


def test_kmeans_map_validates_on_the_host():
    import numpy as np
    from paper_2608_27888_gb300 import ntc
    F = np.zeros((10, 4), dtype=np.float32)
    F[:, 0] = np.arange(10)
    init = np.array([0, 1, 2], dtype=np.uint32)
    out = np.empty(10, dtype=np.uint32)

    def call(F=F, n=10, dim=4, m=3, init=init, iters=5, out=out):
        return ntc._lib.ntc_kmeans_map(F.ctypes.data if F is not None else None, n, dim, m,
                                       init.ctypes.data if init is not None else None, iters,
                                       out.ctypes.data if out is not None else None, None, None)
    assert call(F=None) == ntc.NTC_ERR_INVALID_ARG
    assert call(out=None) == ntc.NTC_ERR_INVALID_ARG
    assert call(m=11) == ntc.NTC_ERR_INVALID_ARG          # more groups than rows
    assert call(m=0) == ntc.NTC_ERR_INVALID_ARG
    assert call(iters=0) == ntc.NTC_ERR_INVALID_ARG
    assert call(dim=0) == ntc.NTC_ERR_INVALID_ARG
    assert call(init=np.array([0, 0, 2], dtype=np.uint32)) == ntc.NTC_ERR_INVALID_ARG  # duplicate start row
    assert call(init=np.array([0, 1, 10], dtype=np.uint32)) == ntc.NTC_ERR_INVALID_ARG  # out of range
    bad = F.copy()
    bad[3, 2] = np.inf
    assert call(F=bad) == ntc.NTC_ERR_INVALID_ARG
    assert b"finite" in ntc._lib.ntc_last_error()


def test_descriptor_layout_matches_the_header(tmp_path):
    """The ctypes ntc_desc has the C struct's fields at the C offsets (a C
    program built against include/ntc.h prints them)."""
    import shutil
    import subprocess
    from paper_2608_27888_gb300 import ntc
    if not shutil.which("gcc"):
        pytest.skip("no C compiler")
    fields = [f for f, _ in ntc.ntc_desc._fields_]
    src = tmp_path / "layout.c"
    body = "\n".join(f'  printf("%zu\\n", offsetof(ntc_desc, {f}));' for f in fields)
    src.write_text("#include <stddef.h>\n#include <stdio.h>\n#include \"ntc.h\"\nint main(void) {\n"
                   + body + '\n  printf("%zu\\n", sizeof(ntc_desc));\n  return 0;\n}\n')
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-std=c99", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)], check=True)
    got = [int(x) for x in subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.split()]
    want = [getattr(ntc.ntc_desc, f).offset for f in fields] + [ctypes.sizeof(ntc.ntc_desc)]
    assert got == want
