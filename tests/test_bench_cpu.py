"""Host logic of bench.py: the source hash that ties a committed ncu
summary to the library code it was taken on."""
import os
import shutil

import bench


def test_strip_comments_keeps_literals_and_collapses_layout():
    src = ('int a = 1; // one\n/* two\n   lines */ const char* s = "//x  /*y*/";\n'
           "char c = '/'; char d = '\\''; const char* e = \"q\\\"//\";\n\n\tint b;")
    out = bench.strip_comments(src)
    assert out == ("int a = 1; const char* s = \"//x  /*y*/\"; char c = '/'; "
                   "char d = '\\''; const char* e = \"q\\\"//\"; int b;")


def test_source_hash_ignores_comments_but_not_code(tmp_path, monkeypatch):
    src = os.path.join(bench.ROOT, "paper_2609_04910_gb300", "csrc")
    root = tmp_path / "repo"
    shutil.copytree(src, root / "paper_2609_04910_gb300" / "csrc",
                    ignore=shutil.ignore_patterns("__pycache__", "*.o", "*.so"))
    monkeypatch.setattr(bench, "ROOT", str(root))
    h0 = bench.kernel_source_hash()
    path = root / "paper_2609_04910_gb300" / "csrc" / "internal.h"
    text = path.read_text()
    path.write_text("// a new comment\n/* and\n   another */\n" + text.replace("\n", "\n\n", 3))
    assert bench.kernel_source_hash() == h0
    path.write_text(text.replace("kFmaMaxChannels = 4", "kFmaMaxChannels = 3", 1))
    assert bench.kernel_source_hash() != h0
