"""The build's staleness check (no compiler run): a library built as the
release variant is not reused when the bounds-checking variant is asked for
(SMEM_DEBUG=1), nor the other way round, and a library without its flavor
stamp or older than a source is rebuilt."""
import os
import time

from paper_2609_32395_gb300 import _build


def _fake_tree(tmp_path, monkeypatch):
    src = tmp_path / "a.cu"
    src.write_text("// source\n")
    lib = tmp_path / "libsmem.so"
    monkeypatch.setattr(_build, "LIB", str(lib))
    monkeypatch.setattr(_build, "_inputs", lambda: [str(src)])
    return src, lib


def _stamp(lib, flavor):
    lib.write_bytes(b"\0")
    (lib.parent / (lib.name + ".flavor")).write_text(flavor + "\n")


def test_flavor_mismatch_forces_a_rebuild(tmp_path, monkeypatch):
    src, lib = _fake_tree(tmp_path, monkeypatch)
    monkeypatch.delenv("SMEM_DEBUG", raising=False)
    assert not _build.up_to_date()  # no library yet
    _stamp(lib, "release")
    later = time.time() + 10
    os.utime(lib, (later, later))
    assert _build.up_to_date()
    monkeypatch.setenv("SMEM_DEBUG", "1")
    assert not _build.up_to_date()  # the checking variant was asked for
    _stamp(lib, "debug")
    os.utime(lib, (later, later))
    assert _build.up_to_date()
    monkeypatch.setenv("SMEM_DEBUG", "0")
    assert not _build.up_to_date()
    _stamp(lib, "release -DX")
    os.utime(lib, (later, later))
    assert _build.up_to_date(extra_flags=("-DX",))
    assert not _build.up_to_date()


def test_missing_stamp_or_newer_source_forces_a_rebuild(tmp_path, monkeypatch):
    src, lib = _fake_tree(tmp_path, monkeypatch)
    monkeypatch.delenv("SMEM_DEBUG", raising=False)
    lib.write_bytes(b"\0")
    later = time.time() + 10
    os.utime(lib, (later, later))
    assert not _build.up_to_date()  # no flavor stamp
    _stamp(lib, "release")
    os.utime(lib, (later, later))
    assert _build.up_to_date()
    os.utime(src, (later + 10, later + 10))
    assert not _build.up_to_date()  # a source newer than the library
