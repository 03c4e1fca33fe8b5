"""Host logic of bench.py that needs no GPU: the source hash that gates each
committed ncu traffic figure follows the code, not its comments, and the
traffic figure is read only while that hash matches; the algorithmic bytes
and flops the roofline lines divide by."""
import os

import numpy as np

import bench


def _tree(tmp_path, text):
    d = tmp_path / "paper_2608_28726_gb300" / "csrc"
    d.mkdir(parents=True, exist_ok=True)
    (d / "k.cu").write_text(text)
    return str(tmp_path)


def test_source_sha_ignores_comments_and_white_space(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "ROOT", _tree(tmp_path, "int f(int x) {\n  return x + 1;\n}\n"))
    a = bench.source_sha(["k.cu"])
    _tree(tmp_path, "// f adds one\nint f(int x) { /* the\n step */ return x + 1;   }\n")
    assert bench.source_sha(["k.cu"]) == a
    _tree(tmp_path, "int f(int x) {\n  return x + 2;\n}\n")
    assert bench.source_sha(["k.cu"]) != a


def test_profiled_traffic_follows_the_source(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "ROOT", _tree(tmp_path, "int g() { return 3; }\n"))
    prof = tmp_path / "p.md"
    prof.write_text("# k\n\n- kernel_source_sha: `%s`\n- dram_bytes_per_launch: `12345`\n"
                    % bench.source_sha(["k.cu"]))
    assert bench.profiled_file_traffic(str(prof), ["k.cu"]) == 12345
    _tree(tmp_path, "int g() { return 4; }\n")
    assert bench.profiled_file_traffic(str(prof), ["k.cu"]) is None
    assert bench.profiled_file_traffic(os.path.join(str(tmp_path), "missing.md"), ["k.cu"]) is None


def test_algorithmic_bytes_of_the_workloads():
    """The bytes behind `roofline.achieved`: per row the logits, the token id
    and the 36-byte record written and read back once (76 bytes beside the
    logits); per request two offsets, 11 aggregates, score, ship and flags (69
    bytes).  The seeded workload shapes give the per-launch figures the
    roofline is quoted on."""
    expect = {"full": (8847, 64, 151936, 2, 2689032372),
              "tiny": (354, 8, 32000, 4, 45339456),
              "wide": (147828, 512, 262144, 4, 155020163184)}
    for name, (rows, reqs, V, eb, total) in expect.items():
        wl = bench.W.make(name)
        assert (wl.n_rows, wl.n_req, wl.vocab, wl.elem_bytes) == (rows, reqs, V, eb), name
        assert bench.algorithmic_bytes(wl) == total, name
        assert total == rows * (V * eb + 76) + reqs * 69, name


def test_head_flops_follow_the_oracle_weight_shapes():
    """The scorer head's algorithmic flops: per layer and token one multiply
    and one add for every entry of the four projection matrices (taken from
    the oracle's weight layout), and per layer, request and head the T x T
    scores and the weighted sum of values over the head width."""
    from oracle import head as oh
    n_layers, lengths = 2, [1, 7, 40]
    p = oh.unpack(np.zeros(oh.n_params(n_layers)), n_layers)
    per_token = sum(2 * p["layers"][0][k].size for k in ("W_qkv", "W_o", "W_1", "W_2"))
    attn = sum(oh.HEADS * 2 * (2 * T * T * oh.DH) for T in lengths)
    step, one_attn = bench.head_flops(lengths, n_layers)
    assert one_attn == attn
    assert step == n_layers * (per_token * sum(lengths) + attn)


def test_quantile_bytes_count_the_weights_of_the_oracle_mlp():
    """One quantile-scorer launch reads each 32-byte record, the offsets and
    the MLP's weights once, and writes score, ship and flags per request."""
    from oracle import quantile as oq
    n_rows, n_req = 1000, 7
    assert bench.qnt_bytes(n_rows, n_req) == (32 * n_rows + 8 * (n_req + 1) + 4 * oq.n_params()
                                              + (4 + 1 + 4) * n_req)


def _oracle_stub(n=3, tau=0.5):
    rng = np.random.Generator(np.random.PCG64(7))
    agg = rng.normal(size=(n, 11))
    score = 1.0 / (1.0 + np.exp(-rng.normal(size=n)))
    return {"agg": agg, "score": score, "ship": (score >= tau).astype(np.uint8),
            "req_flags": np.zeros(n, np.uint32)}


def test_parity_bar_and_value_gate():
    """A stubbed oracle result: outputs equal to it pass; a score off by more
    than 1e-5 + 1e-4 |oracle|, a flipped ship bit outside the 1e-6 band or a
    flag bit fails, and a failing record prints no value."""
    o = _oracle_stub()
    g = {k: v.copy() for k, v in o.items()}
    assert bench.parity_ok(g["agg"], g["score"].astype(np.float32), g["ship"], g["req_flags"],
                           o, 0.5)
    bad = g["score"].copy()
    bad[1] += 2e-5 + 1e-4 * abs(bad[1])
    assert not bench.parity_ok(g["agg"], bad, g["ship"], g["req_flags"], o, 0.5)
    ship = g["ship"].copy()
    ship[0] ^= 1
    assert not bench.parity_ok(g["agg"], g["score"], ship, g["req_flags"], o, 0.5)
    fl = g["req_flags"].copy()
    fl[2] = 1
    assert not bench.parity_ok(g["agg"], g["score"], g["ship"], fl, o, 0.5)
    # a score within 1e-6 of tau may go either way
    o2 = _oracle_stub()
    o2["score"][0] = 0.5 + 5e-7
    o2["ship"][0] = 1
    assert bench.parity_ok(o2["agg"], o2["score"], np.array([0, *o2["ship"][1:]]),
                           o2["req_flags"], o2, 0.5)
    rec = bench.gate_on_parity({"value": 123.0, "parity": {"ok": False}})
    assert rec["value"] is None and "parity" in rec["value_withheld"]
    rec = bench.gate_on_parity({"value": 123.0, "parity": {"ok": True}})
    assert rec["value"] == 123.0 and "value_withheld" not in rec
