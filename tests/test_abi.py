"""The C ABI library builds for sm_103a, loads, and exports exactly the entry
points include/fp8rl.h declares (no GPU needed: nothing is called)."""

import ctypes
import os
import re
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "fp8rl.h")


def _declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(fp8rl_[a-z0-9_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def libpath():
    if shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"):
        pytest.skip("no CUDA toolkit")
    from paper_2609_22870_gb300 import _build
    return _build.build()


def test_header_declares_the_boundary():
    names = _declared()
    for must in ("fp8rl_quantize", "fp8rl_token_logprobs", "fp8rl_calibrate_clip_bounds",
                 "fp8rl_clipped_surrogate", "fp8rl_dlogits_rows", "fp8rl_check"):
        assert must in names


def test_library_exports_every_declared_symbol(libpath):
    lib = ctypes.CDLL(libpath)
    for name in _declared():
        assert hasattr(lib, name), name


def test_no_undeclared_exports(libpath):
    out = subprocess.run(["nm", "-D", "--defined-only", libpath], capture_output=True, text=True).stdout
    exported = sorted(l.split()[-1] for l in out.splitlines() if " T " in l and "fp8rl" in l)
    assert exported == _declared()


def test_header_compiles_as_c(tmp_path):
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no gcc")
    src = tmp_path / "t.c"
    src.write_text('#include "fp8rl.h"\nint main(void){fp8rl_calib_opts o; fp8rl_default_calib_opts(&o);'
                   'return (int)sizeof(fp8rl_calib_result) + (int)sizeof(fp8rl_clip_stats);}\n')
    r = subprocess.run([gcc, "-std=c99", "-Wall", "-Werror", "-c", str(src), "-I",
                        os.path.join(ROOT, "include"), "-o", str(tmp_path / "t.o")],
                       capture_output=True, text=True)
    assert r.returncode == 0, r.stderr


def test_struct_layouts_match_binding(libpath, tmp_path):
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no gcc")
    src = tmp_path / "s.c"
    src.write_text('#include <stdio.h>\n#include "fp8rl.h"\nint main(void){printf("%zu %zu %zu",'
                   'sizeof(fp8rl_calib_opts), sizeof(fp8rl_calib_result), sizeof(fp8rl_clip_stats));}\n')
    exe = tmp_path / "s"
    subprocess.run([gcc, "-std=c99", str(src), "-I", os.path.join(ROOT, "include"), "-o", str(exe)],
                   check=True)
    sizes = [int(x) for x in subprocess.run([str(exe)], capture_output=True, text=True).stdout.split()]
    import importlib.util
    spec = importlib.util.spec_from_file_location("_api_probe", os.path.join(
        ROOT, "paper_2609_22870_gb300", "api.py"))
    api = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(api)  # loads the library; calls nothing on the GPU
    assert sizes == [ctypes.sizeof(api.CalibOpts), ctypes.sizeof(api.CalibResult),
                     ctypes.sizeof(api.ClipStats)]


def test_struct_field_offsets_match_binding(libpath, tmp_path):
    """Every field of the binding's ctypes structs sits at the header's offset
    (the readers and api.n_valid_view index the device buffers by them)."""
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no gcc")
    import importlib.util
    spec = importlib.util.spec_from_file_location("_api_probe2", os.path.join(
        ROOT, "paper_2609_22870_gb300", "api.py"))
    api = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(api)  # loads the library; calls nothing on the GPU
    structs = {"fp8rl_calib_opts": api.CalibOpts, "fp8rl_calib_result": api.CalibResult,
               "fp8rl_clip_stats": api.ClipStats, "fp8rl_clip_diag": api.ClipDiag}
    lines = []
    for cname, cls in structs.items():
        for fname, _ in cls._fields_:
            lines.append(f'printf("{cname}.{fname} %zu\\n", offsetof({cname}, {fname}));')
    src = tmp_path / "o.c"
    src.write_text('#include <stdio.h>\n#include <stddef.h>\n#include "fp8rl.h"\nint main(void){' +
                   "".join(lines) + "return 0;}\n")
    exe = tmp_path / "o"
    subprocess.run([gcc, "-std=c99", str(src), "-I", os.path.join(ROOT, "include"), "-o", str(exe)],
                   check=True)
    got = dict(l.split() for l in subprocess.run([str(exe)], capture_output=True, text=True).stdout.splitlines())
    for cname, cls in structs.items():
        for fname, _ in cls._fields_:
            assert int(got[f"{cname}.{fname}"]) == getattr(cls, fname).offset, (cname, fname)


def test_c_program_links_and_runs(libpath, tmp_path):
    """A plain C consumer links against libfp8rl.so and uses the host-side part
    of the ABI: paper defaults, status strings, size queries and the argument
    checks (every call below returns before any CUDA call)."""
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("no gcc")
    src = tmp_path / "consumer.c"
    src.write_text(r'''
#include <math.h>
#include <stdio.h>
#include <string.h>
#include "fp8rl.h"
#define CHECK(c) do { if (!(c)) { printf("FAIL %s\n", #c); return 1; } } while (0)
int main(void) {
  fp8rl_calib_opts o;
  fp8rl_default_calib_opts(&o);
  CHECK(o.mode == FP8RL_CALIB_EXACT && o.lo_min == 0.5 && o.lo_max == 0.9);
  CHECK(o.hi_min == 1.2 && o.hi_max == 2.0 && o.step == 0.02);
  CHECK(o.delta_lo == 0.05 && o.delta_hi == 0.1 && isnan(o.lo_old) && isnan(o.hi_old));
  for (int s = FP8RL_OK; s <= FP8RL_ETIMEOUT; ++s)
    CHECK(fp8rl_status_string((fp8rl_status)s) != NULL && strlen(fp8rl_status_string((fp8rl_status)s)) > 0);
  CHECK(fp8rl_scales_count(16384, 4096, FP8RL_GRAN_BLOCK, FP8RL_ROLE_ACT) == 16384 * 32);
  CHECK(fp8rl_scales_count(151936, 4096, FP8RL_GRAN_BLOCK, FP8RL_ROLE_WEIGHT) == 1187 * 32);
  CHECK(fp8rl_scales_count(151936, 4096, FP8RL_GRAN_ROWWISE, FP8RL_ROLE_WEIGHT) == 151936);
  CHECK(fp8rl_scales_count(7, 4096, FP8RL_GRAN_TENSOR, FP8RL_ROLE_ACT) == 1);
  CHECK(fp8rl_token_logprobs_workspace_size(16384, 4096, 151936, FP8RL_GRAN_BLOCK) > 0);
  CHECK(fp8rl_lm_head_backward_workspace_size(16384, 4096, 151936) > (size_t)5.7e9);
  /* argument checks: null pointers, bad enums and shapes are refused on the host */
  CHECK(fp8rl_quantize(NULL, 4, 128, 128, FP8RL_GRAN_ROWWISE, FP8RL_ROLE_ACT, NULL, NULL, NULL, 0, NULL)
        == FP8RL_EINVAL);
  CHECK(fp8rl_token_logprobs(NULL, NULL, NULL, NULL, FP8RL_GRAN_BLOCK, 16, 128, 64, NULL, NULL, NULL,
                             NULL, NULL, NULL, 0, NULL) == FP8RL_EINVAL);
  CHECK(fp8rl_calibrate_clip_bounds(NULL, NULL, NULL, NULL, NULL, 10, 0.2f, 0.2f, NULL, NULL, NULL, 0,
                                    NULL) == FP8RL_EINVAL);
  printf("ok\n");
  return 0;
}
''')
    exe = tmp_path / "consumer"
    libdir = os.path.dirname(libpath)
    r = subprocess.run([gcc, "-std=c99", "-Wall", "-Werror", str(src), "-I", os.path.join(ROOT, "include"),
                        "-L", libdir, "-lfp8rl", "-Wl,-rpath," + libdir, "-lm", "-o", str(exe)],
                       capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    run = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert run.returncode == 0 and run.stdout.strip() == "ok", run.stdout + run.stderr


def _prototypes():
    """name -> list of parameter declarations, from the header's prototypes."""
    text = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    out = {}
    for m in re.finditer(r"\b(?:fp8rl_status|size_t|void|uint32_t|int64_t|int|const char\s*\*)\s*(fp8rl_[a-z0-9_]+)\s*\(([^;{]*?)\)\s*;",
                         text, flags=re.S):
        params = [p.strip() for p in m.group(2).split(",")]
        out[m.group(1)] = [] if params == ["void"] else params
    return out


def _ctype_of(param):
    if "*" in param:
        return "ptr"
    base = param.rsplit(None, 1)[0]
    return {"int64_t": "i64", "uint64_t": "u64", "float": "f32", "size_t": "u64", "int": "i32",
            "fp8rl_gran": "i32", "fp8rl_role": "i32", "int32_t": "i32", "fp8rl_status": "i32",
            "fp8rl_calib_mode": "i32"}[base]


def test_binding_signatures_match_the_header(libpath):
    """Every ctypes signature of the Python binding has the header's parameter
    count and kinds (a missing or extra argument would shift every later one)."""
    from paper_2609_22870_gb300 import api
    kinds = {ctypes.c_void_p: "ptr", ctypes.c_int64: "i64", ctypes.c_uint64: "u64", ctypes.c_float: "f32",
             ctypes.c_size_t: "u64", ctypes.c_int: "i32"}  # size_t is uint64 here
    protos = _prototypes()
    for name, (_, args) in api._SIGS.items():
        assert name in protos, name
        want = [_ctype_of(p) for p in protos[name]]
        got = [kinds.get(a, "ptr") for a in args]  # POINTER(struct) types are pointers
        assert got == want, (name, got, want)
