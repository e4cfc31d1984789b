"""CPU checks of the C ABI: the library loads, exports every symbol include/uad.h declares,
and its host-side urgency planner matches the oracle's plan exactly (no GPU needed)."""
import os
import re
from fractions import Fraction

import numpy as np
import pytest

import paper_2609_37772_gb300 as uad
from oracle import plan as P

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_symbols():
    names = set()
    for f in os.listdir(os.path.join(ROOT, "include")):
        if f.endswith(".h"):
            src = open(os.path.join(ROOT, "include", f)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names |= set(re.findall(r"\b(uad_[a-z0-9_]+)\s*\(", src))
    return sorted(names)


def test_library_exports_every_declared_symbol():
    names = declared_symbols()
    assert len(names) >= 12
    for n in names:
        assert hasattr(uad._lib, n), n
    assert set(uad.EXPORTS) <= set(names)
    assert b"sm_103a" in uad.uad_version()


def _oracle_flags(ts):
    return (1 if ts.active else 0) | (2 if ts.ghost and not ts.tau == 1 else 0)


SCHEDULES = [
    [4] * 10 + [7] * 15 + [10] * 25,
    [1] * 4 + [10] * 12,
    [5] * 4 + [10] * 12,
    [3, 1, 4, 1, 5, 9, 2, 6],
    [2] * 16,
    [8, 16, 16, 16],
    [1] * 5,                       # N* = 1: one step, nothing released early
    [64, 1, 33, 64, 2],            # the largest budget the library accepts
]


@pytest.mark.parametrize("budgets", SCHEDULES)
@pytest.mark.parametrize("tr", [True, False])
def test_host_plan_matches_oracle(budgets, tr):
    ns = P.n_star(budgets)
    for k in range(1, ns + 1):
        got_ns, flags, num, den = uad.plan_step(budgets, k, tr)
        assert got_ns == ns
        for i, ts in enumerate(P.step_plan(budgets, k, tr)):
            assert bool(flags[i] & 1) == ts.active
            assert bool(flags[i] & 2) == (ts.ghost and tr)
            assert bool(flags[i] & 16) == (ts.ghost and not tr)
            assert bool(flags[i] & 4) == ts.release
            assert bool(flags[i] & 8) == (int(budgets[i]) < ns)
            assert Fraction(int(num[i]), int(den[i])) == ts.tau
            assert np.gcd(num[i], den[i]) == 1


def test_brute_force_plans():
    """Every budget assignment with H = 3 and budgets 1..4."""
    import itertools
    for b in itertools.product(range(1, 5), repeat=3):
        ns = max(b)
        for k in range(1, ns + 1):
            _, flags, num, den = uad.plan_step(list(b), k, True)
            for i, ts in enumerate(P.step_plan(list(b), k, True)):
                assert Fraction(int(num[i]), int(den[i])) == ts.tau
                assert bool(flags[i] & 4) == ts.release


def test_plan_rejects_bad_budgets():
    with pytest.raises(uad.UADError):
        uad.plan_step([0, 3], 1)
    with pytest.raises(uad.UADError):
        uad.plan_step([65], 1)


STRUCTS = {
    "uad_arch": ["kind", "dtype", "n_layers", "width", "n_heads", "n_kv_heads", "head_dim", "mlp_dim",
                 "action_dim", "chunk_len", "prefix_len", "prefix_width", "rope", "max_batch"],
    "uad_schedule": ["budgets", "batch", "n_exec", "tr", "gac", "chunk_relative", "gac_mask", "rot_dim"],
    "uad_stats": ["evals", "n_star", "nonfinite", "tr_extra_evals"],
    "uad_kernel_stat": ["name", "launches", "pad", "total_ms", "bytes", "flops"],
}
CONSTANTS = ["UAD_OK", "UAD_EINVAL", "UAD_ESTATE", "UAD_ENOMEM", "UAD_ECUDA", "UAD_ETIMEDOUT",
             "UAD_ENONFINITE", "UAD_ETOOBIG", "UAD_KIND_ADARMS", "UAD_KIND_DIT", "UAD_KIND_CONCAT",
             "UAD_DTYPE_F32", "UAD_DTYPE_BF16", "UAD_MAX_STEPS"]


def _cc(tmp_path, src, *extra):
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    c = tmp_path / "prog.c"
    c.write_text(src)
    exe = tmp_path / "prog"
    subprocess.run([cc, "-std=c99", "-pedantic", "-Wall", "-Wextra", "-Werror", "-I",
                    os.path.join(ROOT, "include"), str(c), "-o", str(exe), *extra], check=True)
    return subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout


def test_header_is_plain_c_and_matches_the_binding(tmp_path):
    """include/uad.h compiles as strict C99, and the binding's ctypes structures and constants
    agree with it field by field (sizes and offsets as a C compiler lays them out)."""
    lines = ['#include <stdio.h>', '#include <stddef.h>', '#include "uad.h"', "int main(void) {"]
    for s, fields in STRUCTS.items():
        lines.append(f'  printf("{s} size %zu\\n", sizeof({s}));')
        for f in fields:
            lines.append(f'  printf("{s} {f} %zu\\n", offsetof({s}, {f}));')
    for k in CONSTANTS:
        lines.append(f'  printf("const {k} %d\\n", (int)({k}));')
    lines += ["  return 0;", "}"]
    out = _cc(tmp_path, "\n".join(lines) + "\n")
    got = {}
    for line in out.splitlines():
        a, b, v = line.split()
        got[(a, b)] = int(v)
    import ctypes
    for s, fields in STRUCTS.items():
        cls = getattr(uad, s)
        assert got[(s, "size")] == ctypes.sizeof(cls), s
        assert [f for f, _ in cls._fields_] == fields, s
        for f in fields:
            assert got[(s, f)] == getattr(cls, f).offset, (s, f)
    py = {"UAD_OK": uad.UAD_OK, "UAD_EINVAL": uad.UAD_EINVAL, "UAD_ESTATE": uad.UAD_ESTATE,
          "UAD_ENOMEM": uad.UAD_ENOMEM, "UAD_ECUDA": uad.UAD_ECUDA, "UAD_ETIMEDOUT": uad.UAD_ETIMEDOUT,
          "UAD_ENONFINITE": uad.UAD_ENONFINITE, "UAD_ETOOBIG": uad.UAD_ETOOBIG,
          "UAD_KIND_ADARMS": uad.KIND["adarms"], "UAD_KIND_DIT": uad.KIND["dit"],
          "UAD_KIND_CONCAT": uad.KIND["concat"], "UAD_DTYPE_F32": uad.DTYPE["f32"],
          "UAD_DTYPE_BF16": uad.DTYPE["bf16"], "UAD_MAX_STEPS": uad.MAX_STEPS}
    for k in CONSTANTS:
        assert got[("const", k)] == py[k], k


def test_a_c_program_links_and_plans(tmp_path):
    """A plain C program links against the library and calls its host-only entry points (no GPU):
    the version string and the step plan of a three-group schedule, checked against the oracle."""
    b = [4] * 10 + [7] * 15 + [10] * 25
    src = f"""#include <stdio.h>
#include "uad.h"
int main(void) {{
  const int32_t b[50] = {{{", ".join(map(str, b))}}};
  int32_t f[50], num[50], den[50];
  int k, i;
  printf("%s\\n", uad_version());
  for (k = 1; k <= 10; ++k) {{
    int ns = uad_plan_step(b, 50, k, 1, f, num, den);
    for (i = 0; i < 50; ++i) printf("%d %d %d %d %d %d\\n", ns, k, i, f[i], num[i], den[i]);
  }}
  return 0;
}}
"""
    lib = os.path.dirname(uad.LIB_PATH)
    out = _cc(tmp_path, src, "-L", lib, "-l:libuad.so", "-Wl,-rpath," + lib).splitlines()
    assert "sm_103a" in out[0]
    rows = [list(map(int, line.split())) for line in out[1:]]
    assert len(rows) == 10 * 50
    for ns, k, i, f, num, den in rows:
        ts = P.step_plan(b, k, True)[i]
        assert ns == 10 and bool(f & 1) == ts.active and bool(f & 4) == ts.release
        assert Fraction(num, den) == ts.tau
