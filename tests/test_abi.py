"""The C-ABI library builds, loads and exports every entry point include/tss.h declares (no GPU:
no compute call is made)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    with open(os.path.join(ROOT, "include", "tss.h")) as f:
        src = f.read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(tss_[a-z_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def libtss():
    from paper_2609_26100_gb300 import build
    path = build.build()
    return ctypes.CDLL(path)


def test_header_declares_the_boundary():
    names = _declared()
    for must in ("tss_create", "tss_set_skip_config", "tss_verify", "tss_destroy"):
        assert must in names


def test_library_exports_every_declared_symbol(libtss):
    missing = [n for n in _declared() if not hasattr(libtss, n)]
    assert missing == []


def test_binding_covers_the_exports(libtss):
    from paper_2609_26100_gb300 import native
    assert sorted(native.EXPORTS) == _declared()


def test_status_strings_without_gpu(libtss):
    libtss.tss_status_string.restype = ctypes.c_char_p
    assert libtss.tss_status_string(0) == b"ok"
    assert libtss.tss_status_string(3) == b"KV cache capacity exceeded"


def test_library_built_for_sm103a_only():
    from paper_2609_26100_gb300 import build
    assert build.ARCH == ("-gencode", "arch=compute_103a,code=sm_103a")


def test_header_is_c99_and_a_c_program_links_and_runs(libtss, tmp_path):
    """A plain C program includes the header, takes the address of every declared entry point,
    links against libtss.so and calls tss_status_string (no CUDA call)."""
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    from paper_2609_26100_gb300 import build
    lib = build.build()
    names = _declared()
    src = ["#include \"tss.h\"", "#include <stdio.h>", "#include <string.h>",
           "typedef void (*fnp)(void);",
           "static const fnp table[] = {" + ", ".join(f"(fnp){n}" for n in names) + "};",
           "int main(void) {",
           "  if (strcmp(tss_status_string(TSS_OK), \"ok\") != 0) return 1;",
           "  for (size_t i = 0; i < sizeof(table) / sizeof(table[0]); ++i) if (!table[i]) return 2;",
           "  printf(\"%d\\n\", (int)(sizeof(table) / sizeof(table[0])));",
           "  return 0;",
           "}"]
    c = tmp_path / "abi.c"
    c.write_text("\n".join(src) + "\n")
    exe = tmp_path / "abi"
    libdir = os.path.dirname(lib)
    r = subprocess.run([cc, "-std=c99", "-Wall", "-Wextra", "-Werror", "-I", os.path.join(ROOT, "include"), str(c),
                        "-o", str(exe), "-L", libdir, "-l:libtss.so", f"-Wl,-rpath,{libdir}"],
                       capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    r = subprocess.run([str(exe)], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    assert int(r.stdout) == len(names)


def test_binding_structs_match_the_c_layout(tmp_path):
    """Every ctypes structure of the binding has the size and field offsets that a C compiler gives
    the struct of the same name in tss.h (a field added, dropped or reordered on one side fails)."""
    import shutil
    import subprocess
    from paper_2609_26100_gb300 import native
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    structs = {"tss_arch": native.TssArch, "tss_weights": native.TssWeights, "tss_verify_batch": native.TssVerifyBatch,
               "tss_kv_cache": native.TssKvCache, "tss_verify_result": native.TssVerifyResult,
               "tss_kernel_times": native.TssKernelTimes, "tss_step_bytes": native.TssStepBytes,
               "tss_persistent_plan_info": native.TssPersistentPlanInfo}
    lines = ["#include \"tss.h\"", "#include <stdio.h>", "#include <stddef.h>", "int main(void) {"]
    for cname, py in structs.items():
        lines.append(f"  printf(\"{cname} size %zu\\n\", sizeof({cname}));")
        for fname, _ in py._fields_:
            lines.append(f"  printf(\"{cname} {fname} %zu\\n\", offsetof({cname}, {fname}));")
    lines += ["  return 0;", "}"]
    c = tmp_path / "layout.c"
    c.write_text("\n".join(lines) + "\n")
    exe = tmp_path / "layout"
    r = subprocess.run([cc, "-std=c99", "-Wall", "-Werror", "-I", os.path.join(ROOT, "include"), str(c), "-o", str(exe)],
                       capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split("\n")
    got = {}
    for ln in out:
        if ln:
            cname, field, val = ln.split()
            got[(cname, field)] = int(val)
    for cname, py in structs.items():
        assert got[(cname, "size")] == ctypes.sizeof(py), cname
        for fname, _ in py._fields_:
            assert got[(cname, fname)] == getattr(py, fname).offset, f"{cname}.{fname}"


def test_readme_c_example_compiles(tmp_path):
    """The C example in README.md compiles against tss.h as written."""
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    with open(os.path.join(ROOT, "README.md")) as f:
        text = f.read()
    blocks = re.findall(r"```c\n(.*?)```", text, flags=re.S)
    assert blocks, "README has no C example"
    c = tmp_path / "example.c"
    c.write_text(blocks[0])
    r = subprocess.run([cc, "-std=c99", "-Wall", "-Wextra", "-Werror", "-fsyntax-only", "-I",
                        os.path.join(ROOT, "include"), str(c)], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
