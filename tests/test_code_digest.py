"""The gate of the bench's roofline.traffic: the digest follows the attention
kernel's code, not its comments (bench.code_text_digest)."""
import bench


def test_comment_edits_keep_the_digest():
    a = ('// header\nint f() { return 1; }  // one\n/* block\n   comment */\n'
         'const char *s = "a // b";\n')
    b = '// another header\n// of two lines\nint f() { return 1; }\n\nconst char *s = "a // b";  \n'
    assert bench.code_text_digest(a) == bench.code_text_digest(b)


def test_code_edits_change_the_digest():
    a = 'int f() { return 1; }\n'
    assert bench.code_text_digest(a) != bench.code_text_digest('int f() { return 2; }\n')
    # a changed line structure counts as an edit
    assert bench.code_text_digest(a) != bench.code_text_digest('int f() {\n return 1; }\n')


def test_literals_are_code():
    a = 'const char *s = "x // y"; char c = \'"\';\n'
    b = 'const char *s = "x // z"; char c = \'"\';\n'
    assert bench.code_text_digest(a) != bench.code_text_digest(b)
    # an escaped quote does not end the literal
    assert (bench.code_text_digest('s = "a\\" // b";\n')
            != bench.code_text_digest('s = "a\\" // c";\n'))

