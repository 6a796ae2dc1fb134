"""bench.py's `traffic` figures: the DRAM bytes of one ncu capture, read from the committed
profile summary only while the kernel's sources are the ones that were captured (a changed
kernel reports null, not a stale figure)."""
import hashlib
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402


def _sources_hash(sources):
    h = hashlib.sha256()
    for rel in sources:
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def _profile(tmp_path, nbytes, digest):
    p = tmp_path / "profile.md"
    p.write_text(f"# a kernel\n\n    dram_bytes_per_launch: {nbytes}\n    source_sha256: {digest}\n")
    return str(p)


def test_committed_profiles_carry_the_figures():
    """The summaries in profiles/ hold the machine-read lines (a kernel changed since its
    capture makes the bench report null, which is allowed; a summary without them is not)."""
    import re
    for path in (bench.ATTN_PROFILE, bench.MASK_PROFILE):
        text = open(path).read()
        assert re.search(r"dram_bytes_per_launch:\s*[0-9]+", text), path
        assert re.search(r"source_sha256:\s*[0-9a-f]{64}", text), path


def test_traffic_read_when_the_sources_match(tmp_path):
    digest = _sources_hash(bench.MASK_SOURCES)
    assert bench.profiled_traffic(_profile(tmp_path, 12345, digest), bench.MASK_SOURCES) == 12345


def test_traffic_null_once_a_source_changed(tmp_path):
    stale = "0" * 64
    assert bench.profiled_traffic(_profile(tmp_path, 12345, stale), bench.MASK_SOURCES) is None
    # the attention kernel's hash does not cover the mask kernel's sources
    digest = _sources_hash(bench.ATTN_SOURCES)
    assert bench.profiled_traffic(_profile(tmp_path, 12345, digest), bench.MASK_SOURCES) is None


def test_traffic_null_without_a_summary(tmp_path):
    assert bench.profiled_traffic(str(tmp_path / "missing.md"), bench.MASK_SOURCES) is None
    p = tmp_path / "no_figures.md"
    p.write_text("# a kernel without the machine-read lines\n")
    assert bench.profiled_traffic(str(p), bench.MASK_SOURCES) is None
