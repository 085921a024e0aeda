"""Host-side pieces of bench.py (no GPU): the source hash that decides
whether a committed ncu summary still describes the kernels, and the
profile lookups built on it."""
import os

import bench


def test_code_only_drops_comments_and_keeps_literals():
    src = ('int a = 1;   // one\n'
           '/* block\n   comment */ const char *u = "http://x"; char c = \'/\';\n'
           '\n    f("a\\"b//c");  /* tail */\n')
    assert bench._code_only(src) == ('int a = 1;\n const char *u = "http://x"; char c = \'/\';\n'
                                     'f("a\\"b//c");').replace("\n ", "\n")


def test_comment_edits_keep_the_hash_and_code_edits_change_it(tmp_path, monkeypatch):
    csrc = tmp_path / "paper_2608_20711_gb300" / "csrc"
    csrc.mkdir(parents=True)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    monkeypatch.setattr(bench, "KERNEL_SOURCES", {"k": ("k.cu",)})
    (csrc / "k.cu").write_text("int f() { return 1; }  // one\n")
    h0 = bench.source_hash("k")
    (csrc / "k.cu").write_text("// a new note\n\n    int f() { return 1; }  /* still one */\n")
    h1 = bench.source_hash("k")
    (csrc / "k.cu").write_text("int f() { return 2; }  // one\n")
    h2 = bench.source_hash("k")
    assert h0 == h1 and h0 != h2


def test_committed_profiles_name_every_kernel():
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    for k in bench.KERNEL_SOURCES:
        path = os.path.join(root, "profiles", "%s_batched_gemm_fp16.md" % k)
        assert os.path.exists(path), path


def test_committed_profiles_match_the_kernels_as_built():
    """Every committed ncu summary was taken on its kernel's current code,
    so the bench reports its traffic figure rather than null."""
    for k in bench.KERNEL_SOURCES:
        traffic, path = bench.kernel_traffic(k, "batched_gemm_fp16")
        assert traffic is not None and traffic > 0, (k, path)
