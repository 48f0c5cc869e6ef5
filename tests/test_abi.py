"""The C-ABI library loads and exports every entry point include/*.h declares (CPU)."""
import ctypes
import glob
import os
import re

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_entry_points():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        text = re.sub(r"/\*.*?\*/", "", open(h).read(), flags=re.S)
        names |= set(re.findall(r"\b(estp_[a-z_0-9]+)\s*\(", text))
    return sorted(names)


def test_header_declares_the_path():
    names = declared_entry_points()
    for n in ("estp_token_entropy", "estp_attn_importance", "estp_attn_importance_finalize",
              "estp_pool", "estp_create", "estp_destroy", "estp_attn_lse"):
        assert n in names


def test_library_exports_every_declared_symbol():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_15592_gb300 as estp
    lib = ctypes.CDLL(estp.LIB_PATH)
    missing = [n for n in declared_entry_points() if not hasattr(lib, n)]
    assert not missing, missing
    assert set(estp.EXPORTS) == set(declared_entry_points())


def test_invalid_arguments_rejected_before_any_launch():
    """Host-side validation needs no GPU: a NULL context is refused with INVALID_ARG."""
    import paper_2608_15592_gb300 as estp
    rc = estp.lib.estp_token_entropy(None, None, 1, 4, 8, 8, None, 0, None, None)
    assert rc == estp.ESTP_ERR_INVALID_ARG
    assert b"ctx" in estp.lib.estp_last_error(None)
    rc = estp.lib.estp_attn_importance_finalize(None, 1, None, None)
    assert rc == estp.ESTP_ERR_INVALID_ARG
