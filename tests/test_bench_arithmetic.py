"""The benchmark's byte and rate arithmetic (the roofline's numerator), checked by hand; no GPU."""
import math

import bench
from paper_2604_26412_gb300 import replicas
from paper_2604_26412_gb300 import workloads as wl


def _spec(lens, levels, tree, paged, P=16, hq=32, hkv=8):
    return wl.Spec("t", len(lens), 1, list(lens), list(levels), tree, paged, page_size=P, hq=hq, hkv=hkv, seed=0)


def test_attention_bytes_by_hand():
    # one cache, 100 prefix tokens, 3 draft nodes of which 2 query, paged P = 16, chain
    s = _spec([100], [1, 2], False, True)
    D, hkv, hq = 128, 8, 32
    kv = hkv * (100 + 3) * D * 2 * 2                 # K and V of every visible-key candidate, bf16
    qo = 2 * 1 * 2 * hq * D * 2                      # q in, out out
    lse = 1 * 2 * hq * 4
    pt = math.ceil(100 / 16) * 4
    meta = 1 * 4                                     # seq_lens (no tree parents for a chain)
    assert bench.algorithmic_bytes(s, 3, 2, True) == kv + qo + lse + pt + meta


def test_fp8_target_bytes_halve_only_the_prefix():
    s = _spec([1000, 24], [4, 4], True, False)
    b16 = bench.algorithmic_bytes(s, 8, 4, False)
    b8 = bench.algorithmic_bytes(s, 8, 4, False, target_elem=1)
    # only the prefix K/V shrink: 1024 tokens x 8 heads x 128 dims x (K, V) x 1 byte
    assert b16 - b8 == (1000 + 24) * 8 * 128 * 2
    tree_meta = 2 * 8 * 4
    assert b16 - bench.algorithmic_bytes(_spec([1000, 24], [4, 4], False, False), 8, 4, False) == tree_meta


def test_flops_and_fusion_bytes():
    s = _spec([64], [2], False, True, hq=4, hkv=1)
    assert bench.algorithmic_flops(s, 2, 2) == 4 * 4 * 2 * (64 + 2) * 128
    d, T = 256, 3
    assert bench.fusion_bytes(T, d) == 2 * (4 * d * d + d + 3 * T * d)


def test_whole_job_rate_counts_every_rank_against_the_slowest():
    assert replicas.whole_job_rate(100, steps=10, world=1, max_ms=2.0) == 500_000.0
    assert replicas.whole_job_rate(100, steps=10, world=4, max_ms=2.0) == 2_000_000.0


def test_traffic_records_are_well_formed(tmp_path, monkeypatch):
    """Every committed traffic record has positive DRAM bytes and names an existing profile summary
    and existing kernel sources; the lookup uses a record only while its sources hash to its
    kernel_hash."""
    import json
    import os
    rec = json.load(open(os.path.join(bench.ROOT, "profiles", "traffic.json")))
    csrc = os.path.join(bench.ROOT, "paper_2604_26412_gb300", "csrc")
    assert rec, "no traffic records"
    for key, e in rec.items():
        assert e["dram_bytes_per_call"] > 0, key
        assert os.path.exists(os.path.join(bench.ROOT, e["profile"])), key
        assert len(e["kernel_hash"]) == 16, key
        if key.startswith("w"):  # an attention record names the kernel it was captured on
            assert e.get("kernel") in ("tcgen05", "m16n8k16"), key
        for name in e.get("sources", ()):
            assert os.path.exists(os.path.join(csrc, name)), (key, name)
    # a record is used only while its sources hash to its kernel_hash
    fake_root = tmp_path
    os.makedirs(fake_root / "profiles")
    os.symlink(os.path.join(bench.ROOT, "paper_2604_26412_gb300"), fake_root / "paper_2604_26412_gb300")
    good = {"kernel_hash": bench.kernel_source_hash(bench.MMA_SOURCES), "sources": list(bench.MMA_SOURCES),
            "kernel": "m16n8k16", "dram_bytes_per_call": 123.0, "how": "", "profile": ""}
    stale = dict(good, kernel_hash="0" * 16)
    (fake_root / "profiles" / "traffic.json").write_text(json.dumps({"w5-per_depth": good, "w4-per_depth": stale}))
    monkeypatch.setattr(bench, "ROOT", str(fake_root))
    assert bench.recorded_traffic(5, "per_depth") == 123.0
    assert bench.recorded_traffic(5, "per_depth", kernel="m16n8k16") == 123.0
    assert bench.recorded_traffic(5, "per_depth", kernel="tcgen05") is None  # another kernel ran
    assert bench.recorded_traffic(4, "per_depth") is None
    assert bench.recorded_traffic(3, "per_depth") is None


def test_source_hash_ignores_comments_not_code(tmp_path, monkeypatch):
    import os
    csrc = tmp_path / "paper_2604_26412_gb300" / "csrc"
    os.makedirs(csrc)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    base = 'int f(int a) { return a / 2; }  // halve\nconst char* s = "x // y";\n'
    (csrc / "k.cu").write_text(base)
    h0 = bench.kernel_source_hash(("k.cu",))
    (csrc / "k.cu").write_text("/* header */\n" + base.replace("// halve", "// half of a, it's exact") + "\n\n")
    assert bench.kernel_source_hash(("k.cu",)) == h0            # comments and blank lines only
    (csrc / "k.cu").write_text(base.replace("a / 2", "a / 3"))
    assert bench.kernel_source_hash(("k.cu",)) != h0            # code
    (csrc / "k.cu").write_text(base.replace('"x // y"', '"x // z"'))
    assert bench.kernel_source_hash(("k.cu",)) != h0            # a string literal is code
