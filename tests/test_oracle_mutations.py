"""Mutation check of the oracle's pins: each plausible mistake planted in a copy of the
oracle must make a named pin fail.

For every mutation the oracle package, the pins, their golden fixtures and the workload
generators are copied to a temporary directory, one expression of the copied
oracle/kvlink_oracle.py is replaced, and the named pins run there in a child pytest.
The repository's own files are never modified.  A control run of the same pins on the
unmodified copy must pass, so that a failure means the mutation was caught and not that
the harness is broken.

Not planted: "document tokens also see the prefix".  It changes only document rows of
the training-time map, which are never fresh rows at inference, and which rows a
document token sees beyond its own document is a reading, not something the paper fixes.
"""
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PINS = "tests/test_oracle_pins.py"

# name: (expression in oracle/kvlink_oracle.py, replacement, pins that must catch it)
MUTATIONS = {
    "mask_strict_less": ("<= fresh_pos[:, None]", "< fresh_pos[:, None]",
                         ["test_inference_mask_equals_training_mask_rows"]),
    "rope_sign": ("x1 * c - x2 * s, x2 * c + x1 * s", "x1 * c + x2 * s, x2 * c - x1 * s",
                  ["test_rope_matches_complex_rotation"]),
    "rope_interleaved_pairs": ("x1, x2 = x[..., :h], x[..., h:]", "x1, x2 = x[..., 0::2], x[..., 1::2]",
                               ["test_rope_matches_complex_rotation"]),
    "rope_inv_freq": ("-2.0 * j / np.float64(head_dim)", "-1.0 * j / np.float64(head_dim)",
                      ["test_rope_inv_freq_endpoints"]),
    "gqa_modulo_mapping": ("g = h // G\n", "g = h % Hkv\n",
                           ["test_suffix_attention_matches_bruteforce_training_map"]),
    "score_scale_1_over_D": ("/ np.sqrt(np.float64(D))", "/ np.float64(D)",
                             ["test_score_scale_is_inverse_sqrt_head_dim"]),
    "softmax_wrong_axis": ("p = p / p.sum(axis=1, keepdims=True)", "p = p / p.sum(axis=0, keepdims=True)",
                           ["test_suffix_attention_matches_bruteforce_training_map"]),
    "delta_off_by_one": ("np.full((L, H), s, dtype=np.int64)", "np.full((L, H), s + 1, dtype=np.int64)",
                         ["test_reencode_keys_equal_rotation_at_global_position"]),
    "links_before_document": (
        "        doc_start.append(len(kind))\n        kind += [DOC] * int(L)\n        owner += [i] * int(L)\n"
        "        link_pos.append(list(range(len(kind), len(kind) + n_link)))\n"
        "        kind += [LINK] * n_link\n        owner += [i] * n_link\n",
        "        link_pos.append(list(range(len(kind), len(kind) + n_link)))\n"
        "        kind += [LINK] * n_link\n        owner += [i] * n_link\n"
        "        doc_start.append(len(kind))\n        kind += [DOC] * int(L)\n        owner += [i] * int(L)\n",
        ["test_figure2_layout_and_training_mask"]),
    "fresh_k_v_swapped": ("kb[fp], vb[fp] = k_new, v_new", "kb[fp], vb[fp] = v_new, k_new",
                          ["test_one_document_no_links_is_standard_causal_attention"]),
    "bf16_truncation": ("np.rint(np.ldexp(xf, -q_exp))", "np.trunc(np.ldexp(xf, -q_exp))",
                        ["test_bf16_rounding_matches_torch_on_float32_values"]),
    "paged_blocks_assumed_consecutive": (
        "pool[int(block_table[s + t // block_size]), t % block_size]",
        "pool[int(block_table[s]) + t // block_size, t % block_size]",
        ["test_paged_pool_reads_the_same_documents"]),
    "paged_offset_from_block_start_dropped": (
        "pool[int(block_table[s + t // block_size]), t % block_size]",
        "pool[int(block_table[s + t // block_size]), 0]",
        ["test_paged_pool_reads_the_same_documents"]),
}


def _copy_tree(dst):
    for sub in ("oracle", "workloads", os.path.join("tests", "golden")):
        shutil.copytree(os.path.join(ROOT, sub), os.path.join(dst, sub),
                        ignore=shutil.ignore_patterns("__pycache__", "*.so", "*.o"))
    for f in (PINS, os.path.join("tests", "conftest.py"), "pytest.ini"):
        shutil.copy(os.path.join(ROOT, f), os.path.join(dst, f))


def _run_pins(cwd, names):
    ids = [f"{PINS}::{n}" for n in names]
    env = dict(os.environ, PYTHONPATH=cwd, PYTHONDONTWRITEBYTECODE="1")
    return subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider", *ids],
                          cwd=cwd, env=env, capture_output=True, text=True, timeout=300)


@pytest.fixture(scope="module")
def pristine(tmp_path_factory):
    d = str(tmp_path_factory.mktemp("oracle_copy"))
    _copy_tree(d)
    return d


def test_control_copy_passes_every_named_pin(pristine):
    names = sorted({n for _, _, pins in MUTATIONS.values() for n in pins})
    r = _run_pins(pristine, names)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-2000:]


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_mistake_fails_its_pin(name, pristine, tmp_path):
    before, after, pins = MUTATIONS[name]
    d = str(tmp_path / "mutant")
    shutil.copytree(pristine, d)
    path = os.path.join(d, "oracle", "kvlink_oracle.py")
    src = open(path).read()
    assert src.count(before) >= 1, f"mutation site of {name} not found in the oracle"
    with open(path, "w") as fh:
        fh.write(src.replace(before, after, 1))
    r = _run_pins(d, pins)
    assert r.returncode == 1, f"{name} was not caught by {pins}:\n" + r.stdout[-2000:]
