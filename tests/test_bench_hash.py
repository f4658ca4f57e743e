"""The kernel-code hash that ties committed profile figures to the source they
were taken on: comment and whitespace edits keep it, code edits change it."""
import bench


def test_comments_and_whitespace_do_not_change_the_hash():
    a = 'int f(int x) { return x + 1; }  // one\n/* two */\nconst char *s = "a // b";\n'
    b = '// header\nint   f(int x)\n{\n  return x + 1;  /* inline */\n}\nconst char *s = "a // b";'
    assert bench.code_tokens(a) == bench.code_tokens(b)


def test_code_and_literal_edits_change_the_hash():
    base = 'int f(int x) { return x + 1; } const char *s = "a // b";'
    assert bench.code_tokens(base) != bench.code_tokens(base.replace("x + 1", "x + 2"))
    assert bench.code_tokens(base) != bench.code_tokens(base.replace('"a // b"', '"a /* b"'))
    assert bench.code_tokens("char c = '/'; int d;") == "char c = '/'; int d;"


def test_committed_profiles_match_the_kernel_code():
    for path in (bench.TRAFFIC_FILE, bench.ISSUE_FILE):
        assert bench.profiled(path, "wsgemm8192") is not None, path
