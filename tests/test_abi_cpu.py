"""The C-ABI library on a machine without a GPU: it loads, it exports every
function include/bsm.h declares, argument errors come back as status codes
before any CUDA call, and the host-side scheduler matches the oracle."""
import ctypes
import subprocess

import numpy as np
import pytest

from paper_2002_07062_gb300 import bsm


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__ as g
    g.build()


def test_library_exports_every_header_function():
    names = bsm.header_functions()
    assert len(names) >= 15
    out = subprocess.run(["nm", "-D", "--defined-only", bsm.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    exported = {line.split()[-1] for line in out.splitlines() if line.strip()}
    missing = [n for n in names if n not in exported]
    assert not missing, missing
    for n in names:
        assert hasattr(bsm.lib(), n)


def test_status_strings_and_version():
    assert bsm.status_string(0) == "ok"
    for s in range(1, 9):
        assert bsm.status_string(s) not in ("ok", "unknown status")
    assert bsm.status_string(99) == "unknown status"
    assert bsm.bsm_version() >> 16 == 1


@pytest.mark.parametrize("args,code", [
    ((0, 0, -1, 4, 4, bsm.F32, bsm.POLICY_RR), bsm.ERR_INVALID_ARG),   # B < 0
    ((0, 0, 1, -4, 4, bsm.F32, bsm.POLICY_RR), bsm.ERR_INVALID_ARG),   # R < 0
    ((0, 0, 1, 4, 0, bsm.F32, bsm.POLICY_RR), bsm.ERR_INVALID_ARG),    # C < 1
    ((0, 0, 1, 4, 4, 7, bsm.POLICY_RR), bsm.ERR_INVALID_ARG),          # dtype
    ((0, 0, 1, 4, 4, bsm.F32, 9), bsm.ERR_INVALID_ARG),                # policy
])
def test_argument_errors_without_gpu(args, code):
    rc = bsm.lib().bsm_softmax(*args, None)
    assert rc == code


def test_empty_batch_is_a_no_op():
    assert bsm.lib().bsm_softmax(None, None, 0, 5, 4, bsm.F32, bsm.POLICY_RR, None) == bsm.OK
    assert bsm.lib().bsm_softmax(None, None, 3, 0, 4, bsm.F32, bsm.POLICY_RR, None) == bsm.OK
    assert bsm.lib().bsm_softmax_ragged(None, None, 0, None, None, None, bsm.F32,
                                        bsm.POLICY_RR, 0, None) == bsm.OK


def test_bad_flags_and_null_tables_rejected():
    assert bsm.lib().bsm_softmax_ex(0, 0, 1, 4, 4, bsm.F32, bsm.POLICY_RR, 2, None) == \
        bsm.ERR_INVALID_ARG
    assert bsm.lib().bsm_softmax_ragged(0, 0, 3, None, None, None, bsm.F32, bsm.POLICY_RR, 0,
                                        None) == bsm.ERR_INVALID_ARG
    assert bsm.lib().bsm_plan_create(None, None) == bsm.ERR_INVALID_ARG
    d = bsm.PlanDesc()
    assert bsm.lib().bsm_plan_desc_init(ctypes.byref(d)) == bsm.OK
    assert d.tie_seed == 0x2002070600 and d.lb_weighted == 1 and d.device == -1


def test_schedule_host_rejects_bad_maps():
    with pytest.raises(bsm.BsmError):
        bsm.bsm_schedule_host([(0, 512)], [(256, [0, 5])], 2, 0)      # bank 5 of 2
    with pytest.raises(bsm.BsmError):
        bsm.bsm_schedule_host([(0, 1024)], [(256, [0, 1])], 2, 0)     # past the map
    with pytest.raises(bsm.BsmError):
        bsm.bsm_schedule_host([(0, 512)], [(256, [0, 1])], 2, 0, balance=True, units=[0, 1])


@pytest.mark.parametrize("args,code", [
    ((1, 128, 64, 64, bsm.F32, bsm.POLICY_DYNAMIC), bsm.OK),            # placeholder row
    ((-1, 128, 64, 64, bsm.F32, bsm.POLICY_DYNAMIC), bsm.ERR_INVALID_ARG),
    ((1, 128, 64, 64, 7, bsm.POLICY_DYNAMIC), bsm.ERR_INVALID_ARG),     # output dtype
    ((1, 128, 64, 64, bsm.F32, 9), bsm.ERR_INVALID_ARG),                # policy
    ((1, 64, 64, 64, bsm.F32, bsm.POLICY_DYNAMIC), bsm.ERR_UNSUPPORTED),   # M % 128
    ((1, 128, 96, 64, bsm.F32, bsm.POLICY_DYNAMIC), bsm.ERR_UNSUPPORTED),  # N % 64
    ((1, 128, 64, 80, bsm.F32, bsm.POLICY_DYNAMIC), bsm.ERR_UNSUPPORTED),  # K % 64
    ((1, 128, 64, 0, bsm.F32, bsm.POLICY_DYNAMIC), bsm.ERR_UNSUPPORTED),   # K = 0
])
def test_bmm_argument_errors_without_gpu(args, code):
    B, M, N, K, out, pol = args
    if code == bsm.OK:
        # well-formed but misaligned pointers: rejected before any CUDA call
        rc = bsm.lib().bsm_bmm(0x1008, 0x20000, 0x40000, B, M, N, K, out, pol, None)
        assert rc == bsm.ERR_MISALIGNED
        # output overlapping the first operand
        rc = bsm.lib().bsm_bmm(0x10000, 0x80000, 0x10100, B, M, N, K, out, pol, None)
        assert rc == bsm.ERR_INVALID_ARG
        return
    assert bsm.lib().bsm_bmm(0x10000, 0x80000, 0x100000, B, M, N, K, out, pol, None) == code


def test_bmm_empty_batch_is_a_no_op():
    for B, M, N in [(0, 128, 64), (3, 0, 64), (3, 128, 0)]:
        assert bsm.lib().bsm_bmm(None, None, None, B, M, N, 64, bsm.BF16, bsm.POLICY_RR, None) == bsm.OK


def test_header_is_plain_c_and_links_from_c(tmp_path):
    """include/bsm.h compiles as C11 under -pedantic, and a C program links
    against libbsm.so, gets argument errors back without a GPU, and reads the
    host-only patch table of workload 2 (6144 patches of 32 rows, three
    64 KiB stages) through the C structs."""
    import os
    import shutil
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no C compiler")
    inc = os.path.dirname(bsm.HEADER)
    lib_dir = os.path.dirname(bsm.LIB_PATH)
    src = tmp_path / "capi.c"
    src.write_text(
        "#include <stdio.h>\n#include \"bsm.h\"\n"
        "int main(void) {\n"
        "  int rc = bsm_softmax(NULL, NULL, -1, 4, 4, BSM_F32, BSM_POLICY_DYNAMIC, NULL);\n"
        "  int rb = bsm_bmm(NULL, NULL, NULL, 1, 64, 64, 64, BSM_F32, BSM_POLICY_DYNAMIC, NULL);\n"
        "  static int32_t R[384], C[384];\n"
        "  for (int s = 0; s < 384; ++s) { R[s] = 512; C[s] = 512; }\n"
        "  bsm_plan_desc d;\n"
        "  bsm_plan_desc_init(&d);\n"
        "  d.x = (const void *)(uintptr_t)(1ull << 40); d.y = (void *)(uintptr_t)(1ull << 41);\n"
        "  d.num_slices = 384; d.rows = R; d.cols = C; d.dtype = BSM_F32;\n"
        "  d.policy = BSM_POLICY_DYNAMIC;\n"
        "  bsm_layout lay;\n"
        "  int rl = bsm_plan_layout_host(&d, 152, 232448, NULL, 0, NULL, 0, &lay);\n"
        "  static bsm_patch p[6144];\n"
        "  int rl2 = bsm_plan_layout_host(&d, 152, 232448, p, 6144, NULL, 0, &lay);\n"
        "  int ok = rl == BSM_OK && rl2 == BSM_OK && lay.n_patches == 6144 && lay.n_stages == 3 &&\n"
        "           lay.stage_bytes == 65536 && lay.n_patches_phase1 == 0 && p[1].elem_offset == 32 * 512 &&\n"
        "           p[1].nrows == 32 && p[1].row0 == 32 && p[6143].row0 == 480 && p[6143].slice_rows == 512;\n"
        "  printf(\"%d %d %d %d\\n\", bsm_version(), rc, rb, ok);\n"
        "  return rc == BSM_ERR_INVALID_ARG && rb == BSM_ERR_UNSUPPORTED && ok ? 0 : 1;\n}\n")
    exe = tmp_path / "capi"
    subprocess.run([gcc, "-std=c11", "-Wall", "-Wextra", "-pedantic", "-Werror", "-I", inc, str(src),
                    "-L", lib_dir, "-lbsm", "-Wl,-rpath," + lib_dir, "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True)
    assert out.returncode == 0, out.stdout + out.stderr


def test_plan_create_without_gpu_reports_no_device():
    """A well-formed descriptor reaches the device query (inside the plan's
    trace range, a no-op without a profiler) and comes back as
    BSM_ERR_NO_DEVICE; execute and stats reject a null plan."""
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    d = bsm.PlanDesc()
    assert bsm.lib().bsm_plan_desc_init(ctypes.byref(d)) == bsm.OK
    r = (ctypes.c_int32 * 1)(4)
    c = (ctypes.c_int32 * 1)(64)
    d.x, d.y, d.num_slices = 1 << 40, 1 << 41, 1
    d.rows = ctypes.cast(r, bsm.c_i32p)
    d.cols = ctypes.cast(c, bsm.c_i32p)
    h = ctypes.c_void_p()
    for _ in range(2):
        assert bsm.lib().bsm_plan_create(ctypes.byref(h), ctypes.byref(d)) == bsm.ERR_NO_DEVICE
        assert not h.value
    assert bsm.lib().bsm_plan_execute(None, None) == bsm.ERR_INVALID_ARG
    s = bsm.PlanStats()
    assert bsm.lib().bsm_plan_get_stats(None, ctypes.byref(s)) == bsm.ERR_INVALID_ARG


class _FakeDevTensor:
    """Stands in for a CUDA tensor: the binding only asks where it lives,
    whether it is contiguous, its size and its address."""
    is_cuda = True
    device = "cuda:0"

    def __init__(self, n, es=4, contiguous=True):
        self._n, self._es, self._c = n, es, contiguous

    def is_contiguous(self):
        return self._c

    def numel(self):
        return self._n

    def element_size(self):
        return self._es

    def data_ptr(self):
        return 1 << 40


def test_binding_rejects_host_strided_and_short_tensors():
    """The C ABI sees only addresses, so the binding checks device, layout and
    size before the call; a well-formed call reaches the library (which, on a
    machine without a GPU, answers BSM_ERR_NO_DEVICE)."""
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    F = _FakeDevTensor
    with pytest.raises(ValueError, match="CUDA tensor"):
        bsm.bsm_softmax(torch.zeros(256), F(256), 4, 1, 64, bsm.F32, bsm.POLICY_RR)
    with pytest.raises(ValueError, match="contiguous"):
        bsm.bsm_softmax(F(256), F(256, contiguous=False), 4, 1, 64, bsm.F32, bsm.POLICY_RR)
    with pytest.raises(ValueError, match="needs 1024"):
        bsm.bsm_softmax_ex(F(255), F(256), 4, 1, 64, bsm.F32, bsm.POLICY_RR, 0)
    with pytest.raises(ValueError, match="needs 512"):              # bf16: 2 bytes each
        bsm.bsm_softmax(F(256, es=2), F(255, es=2), 4, 1, 64, bsm.BF16, bsm.POLICY_RR)
    with pytest.raises(ValueError, match="needs"):                  # ragged: the furthest slice
        bsm.bsm_softmax_ragged(F(1000), F(1000), [0, 960], [1, 1], [64, 64], bsm.F32, bsm.POLICY_RR)
    with pytest.raises(ValueError, match="needs"):
        bsm.bsm_softmax_backward(F(256), F(128), F(256), 4, 1, 64, bsm.F32, bsm.POLICY_RR)
    with pytest.raises(ValueError, match="needs"):                  # c: 128 x 64 fp32
        bsm.bsm_bmm(F(128 * 64, es=2), F(64 * 64, es=2), F(128 * 64 - 1), 1, 128, 64, 64,
                    bsm.F32, bsm.POLICY_DYNAMIC)
    with pytest.raises(ValueError, match="needs"):
        bsm.bsm_plan_create(F(100), F(256), [4], [64], bsm.F32, bsm.POLICY_DYNAMIC)
    # well-formed: the call reaches the library
    with pytest.raises(bsm.BsmError) as e:
        bsm.bsm_softmax(F(256), F(256), 4, 1, 64, bsm.F32, bsm.POLICY_RR)
    assert e.value.status == bsm.ERR_NO_DEVICE
    with pytest.raises(bsm.BsmError) as e:
        bsm.bsm_softmax_ragged(F(1024), F(1024), [0, 960], [1, 1], [64, 64], bsm.F32,
                               bsm.POLICY_RR)
    assert e.value.status == bsm.ERR_NO_DEVICE
    # empty batches need no buffer at all
    bsm.bsm_softmax(None, None, 0, 4, 64, bsm.F32, bsm.POLICY_RR)


def test_ragged_extent_host_helper():
    """bsm_ragged_extent: the end of the furthest non-empty slice, 0 for none,
    -1 for a negative offset or column count (host only, no device)."""
    import numpy as np
    from paper_2002_07062_gb300 import bsm

    def ext(off, rows, cols):
        o = np.asarray(off, np.int64)
        r = np.asarray(rows, np.int32)
        c = np.asarray(cols, np.int32)
        return int(bsm.lib().bsm_ragged_extent(len(o), o.ctypes.data_as(bsm.c_i64p),
                                               r.ctypes.data_as(bsm.c_i32p),
                                               c.ctypes.data_as(bsm.c_i32p)))
    assert ext([0, 10], [0, 2], [5, 3]) == 16            # the empty slice is ignored
    assert ext([100, 0], [1, 4], [8, 16]) == 108         # furthest end, not the last slice
    assert ext([], [], []) == 0
    assert ext([0], [0], [7]) == 0
    assert ext([1 << 40], [3], [1 << 20]) == (1 << 40) + 3 * (1 << 20)
    assert ext([-8], [1], [4]) == -1
    assert ext([0], [1], [-4]) == -1
    assert ext([(1 << 63) - 8], [1], [16]) == -1               # past INT64_MAX
