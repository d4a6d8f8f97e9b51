"""The scaffold's test-data helpers for self-contained programs (Sec. 4.1.2),
on the CPU: a host-only probe built with nvcc reads tensor files with
read_binary_file<T> and writes them back with write_binary_file<T>.  A file
is read only as the element type it holds (Sec. 5.2.3's defect becomes an
error), and the compilation tool reports the calling convention the
scaffold's main() emits at compile time."""
import os
import subprocess

import numpy as np
import pytest

import tensor_files as TF
from paper_2609_00058_gb300 import candidate_round as CR
from paper_2609_00058_gb300.build import nvcc

HERE = os.path.dirname(os.path.abspath(__file__))


@pytest.fixture(scope="module")
def probe(tmp_path_factory):
    out = str(tmp_path_factory.mktemp("probe") / "scaffold_io_probe")
    subprocess.check_call([nvcc(), "-O1", "-I" + CR.SCAFFOLD_DIR, "-o", out,
                           os.path.join(HERE, "candidates", "scaffold_io_probe.cu")])
    return out


def run(probe, t, a, b):
    return subprocess.run([probe, t, str(a), str(b)], capture_output=True, text=True)


@pytest.mark.parametrize("dtype,np_t,name", [("f32", np.float32, "float32"), ("u8", np.uint8, "uint8"),
                                             ("i32", np.int32, "int32"), ("bf16", np.uint16, "bfloat16"),
                                             ("f64", np.float64, "float64")])
def test_round_trip(probe, tmp_path, dtype, np_t, name):
    data = np.random.default_rng(1).integers(0, 255, size=6 * 7, dtype=np.uint8).astype(np_t)
    a, b = tmp_path / "a.svt", tmp_path / "b.svt"
    TF.write(a, data, dtype, shape=(6, 7))
    r = run(probe, name, a, b)
    assert r.returncode == 0 and r.stdout.strip() == "42"
    assert open(a, "rb").read() == open(b, "rb").read()
    assert TF.parse(b)[:2] == (dtype, (6, 7))


def test_reading_another_type_is_an_error(probe, tmp_path):
    a = tmp_path / "img.svt"
    TF.write(a, np.arange(16, dtype=np.uint8), "u8")
    r = run(probe, "float32", a, tmp_path / "o.svt")
    assert r.returncode == 3
    assert "element type is uint8, the program reads float32" in r.stderr
    TF.write(a, np.arange(16, dtype=np.int32), "i32")
    r = run(probe, "float32", a, tmp_path / "o.svt")
    assert r.returncode == 3 and "int32" in r.stderr
    assert not os.path.exists(tmp_path / "o.svt")


def test_malformed_files_are_errors(probe, tmp_path):
    a = tmp_path / "bad.svt"
    with open(a, "wb") as f:
        f.write(TF.header("f32", (10,)))
        f.write(bytes(36))  # one element short
    assert run(probe, "float32", a, tmp_path / "o.svt").returncode == 3
    with open(a, "wb") as f:
        f.write(TF.header("f32", (10,)))
        f.write(bytes(44))  # one element too many
    assert run(probe, "float32", a, tmp_path / "o.svt").returncode == 3
    a.write_bytes(np.arange(10, dtype=np.float32).tobytes())  # a headerless file
    r = run(probe, "float32", a, tmp_path / "o.svt")
    assert r.returncode == 3 and "not a tensor file" in r.stderr
    assert run(probe, "float32", tmp_path / "missing.svt", tmp_path / "o.svt").returncode == 3


def test_compile_program_reports_the_calling_convention(tmp_path):
    c = CR.compile_program(os.path.join(HERE, "candidates", "vec_add_inplace.cu"), str(tmp_path))
    assert c.ok and os.path.exists(c.path)
    assert c.calling_convention.startswith("PROGRAM A.svt B.svt OUT.svt [RUNS]")
    assert c.calling_convention.endswith("scratch copy of A")
    bad = CR.compile_program(os.path.join(HERE, "candidates", "vec_add_inplace_broken.cu"), str(tmp_path))
    assert not bad.ok and bad.path is None
