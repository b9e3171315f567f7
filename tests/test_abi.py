"""The C-ABI library: it loads, exports every symbol the header declares, and
rejects bad arguments on the host (no GPU needed: nothing is enqueued)."""
import ctypes
import os
import re

import pytest

from paper_2608_08721_gb300 import binding as lr

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "libraspec.h")


def _declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(libraspec_[a-z_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib():
    from paper_2608_08721_gb300 import build

    build.build()
    return lr.load()


def test_header_declares_the_round_entry_points():
    names = _declared()
    for n in ("libraspec_confidence", "libraspec_select_lengths", "libraspec_verify_attn", "libraspec_accept",
              "libraspec_verify_round", "libraspec_workspace_size", "libraspec_get_status"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    names = _declared()
    assert names
    for n in names:
        assert hasattr(lib, n), "libraspec.so does not export %s" % n
    assert set(names) <= set(lr.SIGNATURES), "binding lacks a signature for %s" % (set(names) - set(lr.SIGNATURES))


def test_version_and_status_strings(lib):
    assert b"sm_103a" in lib.libraspec_version()
    assert lib.libraspec_status_string(-1) == b"invalid argument"


def test_workspace_size_is_host_only_and_validates(lib):
    s = lib.libraspec_workspace_size(64, 32, 128256, 32, 8, 128, 32832)
    assert s > 0 and s % 256 == 0
    assert lib.libraspec_workspace_size(1, 16, 32000, 8, 2, 64, 576) < s
    assert lib.libraspec_workspace_size(1, 16, 32000, 8, 3, 64, 576) == 0      # Hq % Hkv != 0
    # K up to the draft-tree node budget (512) sizes a workspace; beyond, none
    assert lib.libraspec_workspace_size(1, 512, 32000, 8, 2, 64, 576) > 0
    assert lib.libraspec_workspace_size(1, 513, 32000, 8, 2, 64, 576) == 0     # K > max
    assert lib.libraspec_workspace_size(1, 16, 32000, 8, 2, 96, 576) == 0      # head dim


def test_calls_reject_bad_arguments_before_any_launch(lib):
    P = ctypes.c_void_p
    fake = P(0x1000)  # never dereferenced: validation fails first
    assert lib.libraspec_confidence(None, None, None, 1, 2, 8, None, None, None, 0, None) == lr.EINVAL
    assert lib.libraspec_confidence(fake, fake, fake, -1, 2, 8, fake, None, fake, 1 << 20, None) == lr.EINVAL
    assert lib.libraspec_select_lengths(fake, fake, 1, 65, fake, fake, 1 << 20, None) == lr.EINVAL
    assert lib.libraspec_verify_attn(fake, fake, fake, fake, fake, 1, 4, 8, 2, 96, 64, 0.1, fake, None, fake,
                                     1 << 30, None) == lr.EUNSUPPORTED
    assert lib.libraspec_verify_attn(fake, fake, fake, fake, fake, 1, 4, 8, 3, 64, 64, 0.1, fake, None, fake,
                                     1 << 30, None) == lr.EINVAL
    # unaligned K cache pointer
    assert lib.libraspec_verify_attn(fake, P(0x1008), fake, fake, fake, 1, 4, 8, 2, 64, 64, 0.1, fake, None,
                                     fake, 1 << 30, None) == lr.EINVAL
    # workspace too small
    assert lib.libraspec_accept(fake, fake, fake, None, None, fake, fake, 2, 4, 64, 0, 0, 0, fake, fake, fake, 16,
                                None) == lr.EINVAL
    # empty batches are a no-op
    assert lib.libraspec_accept(None, None, None, None, None, None, None, 0, 4, 64, 0, 0, 0, None, None, None, 0,
                                None) == lr.OK


def test_binding_fails_loudly_without_library(monkeypatch, tmp_path):
    monkeypatch.setattr(lr, "_lib", None)
    monkeypatch.setattr(lr, "LIB_PATH", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError, match="not built"):
        lr.load()


def test_newer_entry_points_reject_bad_arguments_before_any_launch(lib):
    P = ctypes.c_void_p
    fake = P(0x1000)  # never dereferenced: validation fails first
    arr = (ctypes.c_void_p * 1)(0x1000)
    # draft trees: node budget above the limit, a missing parent array
    assert lib.libraspec_verify_attn_tree_layers(arr, arr, arr, 1, fake, fake, fake, 1, lr.MAX_TREE_NODES + 1, 8,
                                                 2, 64, 1024, 0.1, arr, None, fake, 1 << 30, None) == lr.EINVAL
    assert lib.libraspec_verify_attn_tree_layers(arr, arr, arr, 1, None, fake, fake, 1, 16, 8, 2, 64, 1024, 0.1,
                                                 arr, None, fake, 1 << 30, None) == lr.EINVAL
    assert lib.libraspec_accept_tree(fake, fake, fake, fake, None, 2, 8, 100, 0, 0, 0, fake, fake, fake, fake,
                                     1 << 30, None) == lr.EINVAL                      # no temperatures
    # the LM head: model dimension not a multiple of 64, a workspace too small, no tokens for probabilities
    assert lib.libraspec_lm_head_stats(fake, fake, None, 1, None, 4, 100, 48, fake, fake, None, fake, 1 << 20,
                                       None) == lr.EUNSUPPORTED
    assert lib.libraspec_lm_head_stats(fake, fake, None, 1, None, 4, 100, 64, fake, fake, None, fake, 16,
                                       None) == lr.EINVAL
    assert lib.libraspec_lm_head_stats(fake, fake, None, 1, None, 4, 100, 64, fake, fake, fake, fake, 1 << 20,
                                       None) == lr.EINVAL
    assert lib.libraspec_lm_head_workspace_size(-1, 100) == 0
    assert lib.libraspec_lm_head_workspace_size(33, 128256) >= 33 * 1002 * 16
    # the KV append: head dim, unaligned source
    assert lib.libraspec_kv_append(fake, arr, arr, 1, fake, 1, 5, 2, 96, 64, fake, 256, None) == lr.EUNSUPPORTED
    assert lib.libraspec_kv_append(P(0x1004), arr, arr, 1, fake, 1, 5, 2, 64, 64, fake, 256, None) == lr.EINVAL
    # confidence + selection without a cost table
    assert lib.libraspec_confidence_select(fake, fake, fake, None, 1, 4, 64, fake, fake, fake, fake, 1 << 20,
                                           None) == lr.EINVAL
    # the staged round without its parts
    args = [None] * 18 + [1, fake] + [1, 4, 64, 8, 2, 64, 64] + [0.1, 0, 0, 0] + [fake] * 6 + [1 << 30, None]
    assert lib.libraspec_verify_round_staged(*args) == lr.EINVAL
    # the bounded-wait self-test: a limit of 0 or above 2 s, a missing flag, a small workspace
    fake256 = P(0x1000)
    assert lib.libraspec_selftest_wait(fake, 0, fake, fake256, 256, None) == lr.EINVAL
    assert lib.libraspec_selftest_wait(fake, 3_000_000_000, fake, fake256, 256, None) == lr.EINVAL
    assert lib.libraspec_selftest_wait(None, 1000, fake, fake256, 256, None) == lr.EINVAL
    assert lib.libraspec_selftest_wait(fake, 1000, fake, fake256, 16, None) == lr.EINVAL
