"""Pins of the pre-scorer oracle (Section 3.1, Eq. 2): an independent
TF-IDF implementation (scikit-learn's vectorizer with its defaults) on ASCII
text, closed forms, and the tokenizer reading on edge cases."""
import math

import numpy as np
import pytest

from oracle import prescore as op

DOCS = [
    b"What is the color of the car in the image? Answer with one word.",
    b"How many people are standing near the red bus_stop sign?",
    b"Describe the image in detail, including the car, the people and the sky.",
    b"Is there a dog? Answer yes or no.",
    b"Read the text on the sign: 'STOP 42' -- what does it say?",
    b"Count the cars. How many cars are red, and how many are blue?",
]


def test_matches_sklearn_tfidf_on_ascii_text():
    sk = pytest.importorskip("sklearn.feature_extraction.text")
    for min_df in (1, 2):
        vec = sk.TfidfVectorizer(min_df=min_df)  # defaults: lowercase, \b\w\w+\b, smooth idf, l2
        X = vec.fit_transform([d.decode() for d in DOCS]).toarray()
        m = op.fit(DOCS, min_df=min_df)
        assert [t.decode() for t in m.terms] == list(vec.get_feature_names_out())
        np.testing.assert_allclose(m.idf, vec.idf_, rtol=0, atol=1e-12)
        prompts = DOCS + [b"the car and the dog and the car", b"nothing known here zzz"]
        Y = vec.transform([p.decode() for p in prompts]).toarray()
        for i, p in enumerate(prompts):
            row, _, _ = op.features(m, p, 0)
            dense = np.zeros(len(m.terms))
            for j, v in row.items():
                dense[j] = v
            np.testing.assert_allclose(dense, Y[i], rtol=0, atol=1e-12)


def test_single_document_corpus_closed_form():
    m = op.fit([b"alpha beta beta gamma"])
    assert m.terms == [b"alpha", b"beta", b"gamma"]
    assert m.idf == [1.0, 1.0, 1.0]  # ln(2 / 2) + 1
    row, img, length = op.features(m, b"Alpha BETA", 3)
    assert row == {0: 1 / math.sqrt(2), 1: 1 / math.sqrt(2)}
    assert (img, length) == (3.0, 2.0)
    row, _, length = op.features(m, b"beta beta beta gamma", 0)
    assert row[1] == pytest.approx(3 / math.sqrt(10), abs=1e-15)
    assert row[2] == pytest.approx(1 / math.sqrt(10), abs=1e-15)
    assert length == 4.0


def test_idf_closed_form():
    # n = 3 documents; "the" in all three, "cat" in one
    m = op.fit([b"the cat", b"the dog", b"the end"])
    j = {t: i for i, t in enumerate(m.terms)}
    assert m.idf[j[b"the"]] == pytest.approx(math.log(4 / 4) + 1)
    assert m.idf[j[b"cat"]] == pytest.approx(math.log(4 / 2) + 1)


def test_out_of_vocabulary_prompt_and_linear_terms():
    m = op.fit([b"alpha beta"])
    w = [0.5, -0.25, 0.75, -0.125]  # alpha, beta, image count, length
    row, img, length = op.features(m, b"gamma delta epsilon", 2)
    assert row == {} and (img, length) == (2.0, 3.0)
    z = op.logit(m, b"gamma delta epsilon", 2, w, 0.1)
    assert z == pytest.approx(0.1 + 0.75 * 2 - 0.125 * 3, abs=1e-15)
    z = op.logit(m, b"alpha", 0, w, 0.0)
    assert z == pytest.approx(0.5 - 0.125, abs=1e-15)  # unit row: alpha = 1


def test_zero_weights_score_one_half():
    m = op.fit(DOCS)
    ps, zs = op.score(m, DOCS, [0, 1, 2, 0, 1, 5], [0.0] * (len(m.terms) + 2), 0.0)
    assert ps == [0.5] * len(DOCS) and zs == [0.0] * len(DOCS)


def test_sigmoid_is_stable_at_large_logits():
    m = op.fit([b"aa"])  # V = 1: w = [aa, image count, length]
    ps, zs = op.score(m, [b"zz", b"zz"], [800, 0], [0.0, 1.0, 0.0], 0.0)
    assert zs == [800.0, 0.0] and ps == [1.0, 0.5]
    ps, zs = op.score(m, [b"zz"], [800], [0.0, -1.0, 0.0], 0.0)
    assert zs == [-800.0] and 0.0 <= ps[0] < 1e-300


def test_tokenizer_reading():
    assert op.tokens(b"It's a C++ test_case, x2 OK!") == [b"it", b"test_case", b"x2", b"ok"]
    # bytes >= 0x80 count as word bytes: a UTF-8 word stays one token
    assert op.tokens("naïve café".encode()) == ["naïve".encode(), "café".encode()]
    assert op.tokens(b"") == [] and op.tokens(b"a b c") == []
