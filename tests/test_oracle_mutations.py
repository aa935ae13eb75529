"""The pins must catch plausible mistakes in the oracle.

Each case plants one mistake (a flipped sign, a dropped term, a wrong index,
a wrong tie-break, ...) in a copy of oracle/ipv_oracle.cpp, builds the copy on
the CPU, and runs the pin suites (test_oracle_pins.py, test_oracle_pool_pins.py,
test_oracle_shared_pins.py, test_oracle_ablation_pins.py) against it. Every
mutant must make that suite fail; the unmutated copy must pass it.
"""
import os
import subprocess
import sys

import pytest

import oracle

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "ipv_oracle.cpp")

MUTANTS = [
    ("TaR sign dropped", "tar[n] = -sum_cos / r;", "tar[n] = sum_cos / r;"),
    ("TaR 1/r dropped", "tar[n] = -sum_cos / r;", "tar[n] = -sum_cos;"),
    ("recent row ignores the patch",
     "n_past + static_cast<int64_t>(t) * p + q", "n_past + static_cast<int64_t>(t) * p"),
    ("recent rows shifted one frame back",
     "n_past + static_cast<int64_t>(t) * p + q", "n_past - p + static_cast<int64_t>(t) * p + q"),
    ("cosine misses the past-key norm",
     "std::max(l2norm(a), eps) * std::max(l2norm(b), eps)", "std::max(l2norm(b), eps)"),
    ("VaN squared norm", "van[n] = l2norm(vv);", "van[n] = dot(vv, vv);"),
    ("VaN scored on keys", "load_row(v, is_bf16, s, cap, D, n, vv);\n      van[n] =",
     "load_row(k, is_bf16, s, cap, D, n, vv);\n      van[n] ="),
    ("all-row VaN squared", "van_out[s * n_tokens + n] = l2norm(vv);",
     "van_out[s * n_tokens + n] = dot(vv, vv);"),
    ("ties go to the higher index", "  return xi < yi;\n}\n\n}  // namespace",
     "  return xi > yi;\n}\n\n}  // namespace"),
    ("lower score wins", "if (xs != ys) return xs > ys;", "if (xs != ys) return xs < ys;"),
    ("alpha|C| rounded up", "std::floor(alpha * ", "std::ceil(alpha * "),
    ("recent frames outside the TaR share", "tar_share - rp)", "tar_share)"),
    ("patch ids ignored", "patch_id ? patch_id[s * cap + n] : n % p", "n % p"),
    ("VaN stage may retake TaR picks", "if (!keep[n]) rest.push_back(n);", "rest.push_back(n);"),
    ("gather copies the wrong row", "s8 + (s * cap_src + n) * row_bytes",
     "s8 + (s * cap_src + j) * row_bytes"),
    ("bf16 widened with the wrong shift", "<< 16;", "<< 15;"),
    ("default r not rounded", "n_frames / 8.0 + 0.5", "n_frames / 8.0"),
    ("recent tokens not kept", "for (int64_t n = n_past; n < n_tokens; ++n) keep[n] = 1;",
     "for (int64_t n = n_past; n + 1 < n_tokens; ++n) keep[n] = 1;"),
    # layer-adaptive VaN pooling
    ("pool mean counts padded positions", "out[n] = acc / static_cast<double>(cnt);",
     "out[n] = acc / static_cast<double>(k * k);"),
    ("pool window one cell too wide", "const int64_t half = k / 2;",
     "const int64_t half = (k + 1) / 2;"),
    ("pool grid rows and columns swapped",
     "const int64_t i = patch[n] / grid_w, j = patch[n] % grid_w;",
     "const int64_t i = patch[n] % grid_h, j = patch[n] / grid_h;"),
    ("CV with the sample standard deviation", "std::sqrt(ss / static_cast<double>(count))",
     "std::sqrt(ss / static_cast<double>(count - 1))"),
    ("CV of one head instead of the layer", "const int64_t count = n_kv_heads * n_tokens;",
     "const int64_t count = n_tokens;"),
    ("pool-size threshold inclusive", "if (cv < tau[0]) return 7;", "if (cv <= tau[0]) return 7;"),
    ("frames of a fresh cache merged", "static_cast<int64_t>(frame_id[s * id_stride + n]) : n / p;",
     "static_cast<int64_t>(frame_id[s * id_stride + n]) : 0;"),
    ("frame ids ignored", "frame[n] = patch_id ? static_cast<int64_t>(frame_id[s * id_stride + n])",
     "frame[n] = patch_id ? static_cast<int64_t>(0)"),
    ("CV without the recent frames", "if (oracle_van_pool(all.data(),",
     "if (oracle_van_pool(van.data(),"),
    ("selection ranks raw VaN", "tau, van.data(), pool_size_out,",
     "tau, all.data(), pool_size_out,"),
    # per-layer shared index set
    ("shared blocks hold only the first head", "  for (int h = 0; h < H; ++h) {\n    load_row(base, is_bf16, l * H + h, cap, D, n, row);",
     "  for (int h = 0; h < 1; ++h) {\n    load_row(base, is_bf16, l * H + h, cap, D, n, row);"),
    ("shared layer reads another layer's heads", "load_row(base, is_bf16, l * H + h, cap, D, n, row);",
     "load_row(base, is_bf16, l + h, cap, D, n, row);"),
    ("shared compaction uses the head's own index row",
     "kept_slab[s * budget + j] = kept_sel[(s / H) * budget + j];",
     "kept_slab[s * budget + j] = kept_sel[(s % H) * budget + j];"),
    # ablation variants
    ("TaR Reverse does not reverse", "for (double& x : tar) x = -x;", "for (double& x : tar) x = x;"),
    ("VaN Reverse reverses TaR", "for (double& x : van) x = -x;", "for (double& x : tar) x = -x;"),
    ("frame mean over the whole slab",
     "frame[n] = frame_id ? static_cast<int64_t>(frame_id[u * id_stride + n]) : n / p;",
     "frame[n] = frame_id ? static_cast<int64_t>(frame_id[u * id_stride + n]) : 0;"),
    ("frame mean divides by the frame size p", "t[n] = a.first / static_cast<double>(a.second);",
     "t[n] = a.first / static_cast<double>(p);"),
    ("uniform frames counted from the oldest", "frames.push_back(F - 1 - (i * F) / k);",
     "frames.push_back((i * F) / k);"),
    ("uniform interval rounded up", "frames.push_back(F - 1 - (i * F) / k);",
     "frames.push_back(F - 1 - (i * F + k - 1) / k);"),
    ("uniform keeps the first row of each frame only", "kept[j++] = static_cast<int32_t>(f * p + q);",
     "kept[j++] = static_cast<int32_t>(f * p);"),
    ("frame ids of a fresh cache compacted as patch ids",
     "src_fid ? src_fid[s * cap_src + n] : static_cast<uint32_t>(n / p)",
     "src_fid ? src_fid[s * cap_src + n] : static_cast<uint32_t>(n % p)"),
]


def _run_pins_with(lib_path: str) -> int:
    env = dict(os.environ, IPV_ORACLE_LIB_OVERRIDE=lib_path)
    cmd = [sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider",
           os.path.join(ROOT, "tests", "test_oracle_pins.py"),
           os.path.join(ROOT, "tests", "test_oracle_pool_pins.py"),
           os.path.join(ROOT, "tests", "test_oracle_shared_pins.py"),
           os.path.join(ROOT, "tests", "test_oracle_ablation_pins.py")]
    return subprocess.run(cmd, env=env, cwd=ROOT, capture_output=True, timeout=300).returncode


def _build_variant(tmp_path, name: str, text: str) -> str:
    src = tmp_path / f"{name}.cpp"
    src.write_text(text)
    out = str(tmp_path / f"lib{name}.so")
    subprocess.run(oracle.build_cmd(str(src), out), check=True)
    return out


def test_unmutated_copy_passes(tmp_path):
    with open(SRC) as fh:
        text = fh.read()
    assert _run_pins_with(_build_variant(tmp_path, "clean", text)) == 0


@pytest.mark.parametrize("name,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_mutant_is_caught(tmp_path, name, old, new):
    with open(SRC) as fh:
        text = fh.read()
    # A line the per-head and the shared-head scoring share is mutated in both.
    assert text.count(old) >= 1, f"mutation anchor not present: {old!r}"
    lib = _build_variant(tmp_path, "mutant", text.replace(old, new))
    assert _run_pins_with(lib) != 0, f"pins did not catch: {name}"
