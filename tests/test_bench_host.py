"""bench.py's bookkeeping on the host (no GPU): the key that ties a committed
ncu traffic record to the attention kernel's code, and the record lookup."""
import json

import bench


def test_code_key_ignores_comments_but_not_code(tmp_path):
    src = open(bench.ATTN_SRC, encoding="utf-8").read()
    same = tmp_path / "comments.cu"
    same.write_text(src.replace("// ", "// (edited) ", 7) + "\n// a trailing note\n\n")
    changed = tmp_path / "code.cu"
    assert "constexpr int kVJobs = 2 * kStages;" in src
    changed.write_text(src.replace("constexpr int kVJobs = 2 * kStages;",
                                   "constexpr int kVJobs = 3 * kStages;"))
    key = bench.attn_code_key()
    assert len(key) == 16 and key == bench.attn_code_key(str(same))
    assert bench.attn_code_key(str(changed)) != key


def test_traffic_record_scales_only_for_the_same_code(tmp_path):
    rec = {"attn_code_key": bench.attn_code_key(), "traffic_over_algorithmic": 1.25}
    (tmp_path / "attn_traffic_cfg7.json").write_text(json.dumps(rec))
    assert bench._committed_traffic(7, 1000, profiles=str(tmp_path)) == 1250
    rec["attn_code_key"] = "0" * 16
    (tmp_path / "attn_traffic_cfg7.json").write_text(json.dumps(rec))
    assert bench._committed_traffic(7, 1000, profiles=str(tmp_path)) is None
    assert bench._committed_traffic(8, 1000, profiles=str(tmp_path)) is None  # no record


def test_committed_records_carry_a_code_key():
    for cfg in (1, 2, 3, 4):
        rec = json.load(open(f"{bench.ROOT}/profiles/attn_traffic_cfg{cfg}.json"))
        assert len(rec["attn_code_key"]) == 16
        assert 1.0 <= rec["traffic_over_algorithmic"] < 1.1
