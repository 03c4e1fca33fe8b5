"""The prompt pre-scorer (Section 3.1, Eq. 2) in the library against the
float64 oracle.  It runs on the host CPU, as the paper keeps it off the
accelerator, so these tests need no GPU; they call the C ABI through the
binding."""
import numpy as np
import pytest

from oracle import prescore as op


@pytest.fixture(scope="module")
def B():
    from paper_2608_28726_gb300 import build
    build.build()
    from paper_2608_28726_gb300 import binding
    return binding


@pytest.fixture(scope="module")
def corpus():
    from paper_2608_28726_gb300 import workloads as W
    docs, _ = W.prompts(600, seed=9201)
    prompts, images = W.prompts(300, seed=9202)
    return docs, prompts, images


@pytest.mark.parametrize("min_df", [1, 2, 5])
def test_vocabulary_and_features_match_the_oracle(B, corpus, min_df):
    docs, prompts, _ = corpus
    m = op.fit(docs, min_df=min_df)
    ps = B.pr_prescorer_fit(docs, min_df=min_df)
    try:
        V = B.pr_prescorer_vocab_size(ps)
        assert V == len(m.terms)
        assert [B.pr_prescorer_term(ps, j) for j in range(V)] == m.terms
        assert B.pr_prescorer_term(ps, V) is None and B.pr_prescorer_term(ps, -1) is None
        for p in prompts[:120] + [b"", b"a b c", b"Zzzz qqqq"]:
            cols, vals, length = B.pr_prescorer_features(ps, p)
            row, _, olen = op.features(m, p, 0)
            assert length == olen
            assert cols.tolist() == sorted(row)
            np.testing.assert_allclose(vals, [row[j] for j in sorted(row)], rtol=1e-6, atol=1e-7)
    finally:
        B.pr_prescorer_destroy(ps)


def test_scores_match_the_oracle(B, corpus):
    from paper_2608_28726_gb300 import workloads as W
    docs, prompts, images = corpus
    m = op.fit(docs, min_df=2)
    ps = B.pr_prescorer_fit(docs, min_df=2)
    try:
        w, b = W.prescore_weights(B.pr_prescorer_vocab_size(ps))
        p_lib, z_lib = B.pr_prescorer_score(ps, prompts, images, w, b)
        p_or, z_or = op.score(m, prompts, images, w.astype(np.float64), b)
        # float32 outputs of double sums
        np.testing.assert_allclose(z_lib, z_or, rtol=1e-6, atol=1e-5)
        np.testing.assert_allclose(p_lib, p_or, rtol=0, atol=1e-6)
        assert np.ptp(np.asarray(p_or)) > 0.1  # the weights separate the prompts
    finally:
        B.pr_prescorer_destroy(ps)


def test_thread_count_does_not_change_results(B, corpus):
    from paper_2608_28726_gb300 import workloads as W
    docs, prompts, images = corpus
    ps = B.pr_prescorer_fit(docs)
    try:
        w, b = W.prescore_weights(B.pr_prescorer_vocab_size(ps), seed=9301)
        ref = B.pr_prescorer_score(ps, prompts, images, w, b, n_threads=1)
        for nt in (2, 3, 7, 0, 1000):
            got = B.pr_prescorer_score(ps, prompts, images, w, b, n_threads=nt)
            assert np.array_equal(got[0], ref[0]) and np.array_equal(got[1], ref[1])
    finally:
        B.pr_prescorer_destroy(ps)


def test_edge_cases(B):
    ps = B.pr_prescorer_fit([b"alpha beta beta gamma", "naïve café".encode()])
    try:
        V = B.pr_prescorer_vocab_size(ps)
        m = op.fit([b"alpha beta beta gamma", "naïve café".encode()])
        assert V == len(m.terms) == 5
        w = np.arange(V + 2, dtype=np.float32) * 0.25 - 0.5
        prompts = [b"", b"a", "Café? NAÏVE!".encode(), b"alpha " * 50, b"unknown words only"]
        imgs = [0, 3, 1, 0, 2]
        p_lib, z_lib = B.pr_prescorer_score(ps, prompts, imgs, w, 0.25, n_threads=2)
        p_or, z_or = op.score(m, prompts, imgs, w.astype(np.float64), 0.25)
        np.testing.assert_allclose(z_lib, z_or, rtol=1e-6, atol=1e-6)
        np.testing.assert_allclose(p_lib, p_or, rtol=0, atol=1e-7)
        # no prompts: nothing to do
        s, z = B.pr_prescorer_score(ps, [], [], w, 0.0)
        assert s.size == 0 and z.size == 0
        # a vocabulary from an empty corpus: only the image count and length count
        ps0 = B.pr_prescorer_fit([])
        assert B.pr_prescorer_vocab_size(ps0) == 0
        s, z = B.pr_prescorer_score(ps0, [b"two words"], [1], np.array([0.5, 0.25], np.float32),
                                    0.0)
        assert z[0] == pytest.approx(0.5 + 0.5)
        B.pr_prescorer_destroy(ps0)
    finally:
        B.pr_prescorer_destroy(ps)


def test_bad_arguments(B):
    ps = B.pr_prescorer_fit([b"alpha beta"])
    try:
        w = np.zeros(4, np.float32)
        with pytest.raises(B.PRError):
            B.pr_prescorer_score(ps, [b"alpha"], [-1], w, 0.0)
        with pytest.raises(B.PRError):
            B.pr_prescorer_score(ps, [b"alpha"], [0], np.zeros(3, np.float32), 0.0)
        with pytest.raises(B.PRError):
            B.pr_prescorer_score(ps, [b"al\x00pha"], [0], w, 0.0)
        with pytest.raises(B.PRError):
            B.pr_prescorer_fit([b"x"], min_df=0)
        with pytest.raises(B.PRError):  # the row does not fit the given capacity
            B.pr_prescorer_features(ps, b"alpha beta", cap=1)
    finally:
        B.pr_prescorer_destroy(ps)


def test_text_marshalling(B):
    """The prompts reach the C call as NUL-terminated strings in one buffer,
    addressed by a pointer array: str, bytes and non-ASCII text read back as
    given; a NUL inside a text is refused."""
    import ctypes
    texts = ["plain text", b"raw bytes \xff\xfe", "naïve café", "", b"", "x" * 5000]
    buf, ptrs, n = B._texts(texts)
    assert n == len(texts) and ptrs.dtype == np.uint64
    for t, p in zip(texts, ptrs):
        want = t.encode() if isinstance(t, str) else t
        assert ctypes.string_at(int(p)) == want
    buf, ptrs, n = B._texts(["only", "strings"])
    assert [ctypes.string_at(int(p)) for p in ptrs] == [b"only", b"strings"]
    buf, ptrs, n = B._texts([])
    assert n == 0
    for bad in (["a\0b"], [b"a", b"\0"], ["ok", "no\0"]):
        with pytest.raises(B.PRError):
            B._texts(bad)


def test_long_tokens_and_many_terms(B):
    """Tokens longer than the scan's first buffer (64 bytes) and a corpus with
    thousands of distinct terms (the fitting table grows several times)."""
    long_a = b"a" * 300
    long_b = b"Tok" + b"x" * 5000 + b"end"
    docs = [b"w%05d common" % i for i in range(5000)] + [long_a + b" " + long_b, long_a]
    ps = B.pr_prescorer_fit(docs, min_df=1)
    try:
        m = op.fit(docs, min_df=1)
        V = B.pr_prescorer_vocab_size(ps)
        assert V == len(m.terms) == 5000 + 3
        assert [B.pr_prescorer_term(ps, j) for j in (0, V - 1)] == [m.terms[0], m.terms[-1]]
        for p in (long_a, long_b + b" " + long_a + b" w00042", b"COMMON " + long_b.upper()):
            cols, vals, length = B.pr_prescorer_features(ps, p)
            row, _, olen = op.features(m, p, 0)
            assert length == olen and cols.tolist() == sorted(row)
            np.testing.assert_allclose(vals, [row[j] for j in sorted(row)], rtol=1e-6, atol=1e-7)
    finally:
        B.pr_prescorer_destroy(ps)
