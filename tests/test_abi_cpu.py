"""CPU checks of the C ABI: the library loads, exports every function the
header declares, and rejects bad arguments on the host before any CUDA call.
No kernel runs here."""
import ctypes as C
import os
import re

import pytest
import torch

import paper_2606_26631_gb300 as prcr
from paper_2606_26631_gb300 import _binding as B

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    src = open(os.path.join(ROOT, "include", "prcr.h")).read()
    return sorted(set(re.findall(r"PRCR_API\s+[\w\s\*]+?\b(prcr_\w+)\s*\(", src)))


def test_header_declares_the_exports():
    assert _declared() == sorted(prcr.EXPORTS)


def test_library_exports_every_declared_symbol():
    L = prcr.lib()
    for name in _declared():
        assert hasattr(L, name), name
    assert prcr.version() == 2


def test_header_constants_match_binding():
    src = open(os.path.join(ROOT, "include", "prcr.h")).read()
    consts = dict(re.findall(r"#define (PRCR_\w+)\s+(-?\d+)u?\b", src))
    for name, val in (("PRCR_OK", B.OK), ("PRCR_EINVAL", B.EINVAL), ("PRCR_EALIGN", B.EALIGN),
                      ("PRCR_EWORKSPACE", B.EWORKSPACE), ("PRCR_ECUDA", B.ECUDA),
                      ("PRCR_ST_IDX_RANGE", B.ST_IDX_RANGE), ("PRCR_ST_NO_BLOCK", B.ST_NO_BLOCK),
                      ("PRCR_ST_CAPACITY", B.ST_CAPACITY), ("PRCR_ST_CSR", B.ST_CSR),
                      ("PRCR_ST_POS_RANGE", B.ST_POS_RANGE), ("PRCR_MODE_PCR", B.MODE_PCR),
                      ("PRCR_MODE_ORIGINAL", B.MODE_ORIGINAL), ("PRCR_MODE_UIR", B.MODE_UIR),
                      ("PRCR_MODE_LPA", B.MODE_LPA), ("PRCR_CACHE_PAGED", B.CACHE_PAGED),
                      ("PRCR_LAYOUT_INTERLEAVED", B.LAYOUT_INTERLEAVED),
                      ("PRCR_FLAG_DEGENERATE_CENTER", B.FLAG_DEGENERATE_CENTER)):
        assert int(consts[name]) == val, name
    # struct layouts: ctypes sizes equal what the C compiler lays out (checked by offsets)
    assert C.sizeof(B.RopeCfg) == 40
    assert C.sizeof(B.StoreDesc) == 64
    assert C.sizeof(B.CacheDesc) == 80
    assert C.sizeof(B.RevisitBatch) == 56
    assert C.sizeof(B.Outputs) == 40


def test_next_text_pos_and_workspace():
    assert prcr.next_text_pos(200, 16, prcr.MODE_PCR) == 201
    assert prcr.next_text_pos(200, 16, prcr.MODE_ORIGINAL) == 201
    assert prcr.next_text_pos(200, 16, prcr.MODE_UIR) == 201
    assert prcr.next_text_pos(200, 16, prcr.MODE_LPA) == 217
    assert prcr.next_text_pos(200, 16, 9) == -(2 ** 63)
    assert prcr.workspace_size(0) == 0
    assert prcr.workspace_size(1) >= 40
    assert prcr.workspace_size(1000) >= 40 * 1000
    assert prcr.lib().prcr_error_string(-3) == b"workspace missing or too small"


# ----------------------------------------------------------------------------
# host-side validation (fake, aligned device addresses: never dereferenced,
# since every case below is rejected before any CUDA call)
# ----------------------------------------------------------------------------
FAKE = 1 << 40


def _descs(**over):
    cfg = prcr.rope_cfg(2, 2, 64, (8, 12, 12))
    st = B.StoreDesc(k=FAKE, v=FAKE + 4096, coords=FAKE + 8192, seq_stride=2 * 64 * 128,
                     layer_stride=64 * 128, token_stride=128, coord_seq_stride=192, n_seqs=1,
                     n_tokens=64)
    ca = B.CacheDesc(kind=0, block_size=1, k=FAKE + 65536, v=FAKE + 131072, seq_stride=2 * 256 * 128,
                     layer_stride=256 * 128, block_stride=0, slot_stride=128, block_table=None,
                     bt_stride=0, n_blocks=0, max_slots=256, n_seqs=1)
    ba = B.RevisitBatch(seq_rev_off=FAKE + 2 ** 20, rev_tok_off=FAKE + 2 ** 20 + 64,
                        idx=FAKE + 2 ** 20 + 128, p_txt=FAKE + 2 ** 20 + 256,
                        cache_len_in=FAKE + 2 ** 20 + 512, n_seqs=1, n_revisits=1, total_k=16)
    ou = B.Outputs(cache_len_out=FAKE + 2 ** 21, next_pos_out=FAKE + 2 ** 21 + 64, pos_out=None,
                   slot_out=None, status=FAKE + 2 ** 21 + 128)
    args = dict(cfg=cfg, st=st, ca=ca, ba=ba, ou=ou, mode=0, L=2, flags=0, ws=FAKE + 2 ** 22,
                ws_bytes=prcr.workspace_size(16))
    for k, v in over.items():
        if "." in k:
            obj, field = k.split(".")
            setattr(args[obj], field, v)
        else:
            args[k] = v
    return args


def _call(name="prcr_rebind_inject", **over):
    a = _descs(**over)
    return getattr(prcr.lib(), name)(C.byref(a["cfg"]), C.byref(a["st"]), C.byref(a["ca"]),
                                     C.byref(a["ba"]), C.byref(a["ou"]), a["mode"], a["L"],
                                     a["flags"], a["ws"], a["ws_bytes"], None)


BAD = [
    ({"cfg.head_dim": 40}, B.EINVAL),            # not a multiple of 16
    ({"cfg.head_dim": 512}, B.EINVAL),           # above the maximum
    ({"cfg.n_layers": 0}, B.EINVAL),
    ({"cfg.layout": 7}, B.EINVAL),
    ({"cfg.theta": 1.0}, B.EINVAL),
    ({"cfg.reserved": 1}, B.EINVAL),
    ({"cfg.n_kv_heads": 64, "cfg.head_dim": 256}, B.EINVAL),  # row above 8192 elements
    ({"st.k": None}, B.EINVAL),
    ({"st.token_stride": 64}, B.EINVAL),         # shorter than a row
    ({"st.k": FAKE + 8}, B.EALIGN),
    ({"st.layer_stride": 64 * 128 + 4}, B.EALIGN),
    ({"ca.kind": 5}, B.EINVAL),
    ({"ca.v": FAKE + 2}, B.EALIGN),
    ({"ca.slot_stride": 100}, B.EINVAL),
    ({"ca.kind": 1, "ca.block_table": None}, B.EINVAL),
    ({"ca.kind": 1, "ca.block_table": FAKE + 2, "ca.block_size": 16}, B.EALIGN),
    ({"mode": 4}, B.EINVAL),
    ({"L": -1}, B.EINVAL),
    ({"flags": 2}, B.EINVAL),
    ({"ba.n_seqs": 2}, B.EINVAL),                # more sequences than the store holds
    ({"ba.total_k": -1}, B.EINVAL),
    ({"ba.total_k": 2 ** 31}, B.EINVAL),
    ({"ba.idx": None}, B.EINVAL),
    ({"ba.p_txt": FAKE + 4}, B.EALIGN),
    ({"ou.status": None}, B.EINVAL),
    ({"ou.cache_len_out": FAKE + 2 ** 20 + 512}, B.EINVAL),  # aliases cache_len_in
    ({"ws": None}, B.EWORKSPACE),
    ({"ws_bytes": 64}, B.EWORKSPACE),
    ({"ws": FAKE + 2 ** 22 + 8}, B.EALIGN),
]


@pytest.mark.parametrize("over,code", BAD, ids=[",".join(o) for o, _ in BAD])
@pytest.mark.parametrize("entry", ["prcr_rebind_inject", "prcr_plan", "prcr_rebind_apply"])
def test_host_validation(entry, over, code):
    assert _call(entry, **over) == code


def test_empty_batch_is_a_no_op():
    # n_seqs == 0 with nothing selected: accepted, nothing launched
    assert _call(**{"ba.n_seqs": 0, "ba.n_revisits": 0, "ba.total_k": 0}) == B.OK
    assert _call(**{"ba.n_seqs": 0, "ba.n_revisits": 1, "ba.total_k": 0}) == B.EINVAL


def test_store_raw_validation():
    a = _descs()
    L = prcr.lib()

    def call(seq=0, l0=0, nl=2, m0=0, mc=4, k=FAKE + 2 ** 23, v=FAKE + 2 ** 24, ls=4 * 128, ts=128,
             coords=None):
        return L.prcr_store_raw(C.byref(a["cfg"]), C.byref(a["st"]), seq, l0, nl, m0, mc, k, v, ls,
                                ts, coords, None)

    assert call(seq=1) == B.EINVAL
    assert call(l0=1, nl=2) == B.EINVAL
    assert call(m0=62, mc=4) == B.EINVAL
    assert call(k=None) == B.EINVAL
    assert call(k=FAKE + 2 ** 23 + 2) == B.EALIGN
    assert call(ts=100) == B.EINVAL
    assert call(nl=0) == B.OK and call(mc=0) == B.OK  # nothing to copy


def test_binding_type_checks():
    k = torch.zeros(1, 2, 8, 2, 64, dtype=torch.float16)
    with pytest.raises(TypeError):
        prcr.store_desc(k, k, torch.zeros(1, 8, 3, dtype=torch.int32))
    with pytest.raises(TypeError):
        prcr.revisit_batch(torch.zeros(2, dtype=torch.int64), torch.zeros(2, dtype=torch.int32),
                           torch.zeros(1, dtype=torch.int32), torch.zeros(1, dtype=torch.int64),
                           torch.zeros(1, dtype=torch.int32))


def test_struct_layout_matches_c_compiler(tmp_path):
    """Compile a tiny C program against include/prcr.h and compare every
    field offset and struct size with the ctypes mirror."""
    import shutil
    import subprocess
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    structs = {"prcr_rope_cfg": B.RopeCfg, "prcr_store_desc": B.StoreDesc,
               "prcr_cache_desc": B.CacheDesc, "prcr_revisit_batch": B.RevisitBatch,
               "prcr_outputs": B.Outputs}
    lines = ["#include <stdio.h>", "#include <stddef.h>", '#include "prcr.h"', "int main(void){"]
    for cname, py in structs.items():
        lines.append(f'printf("{cname} size %zu\\n", sizeof({cname}));')
        for f, _ in py._fields_:
            lines.append(f'printf("{cname} {f} %zu\\n", offsetof({cname}, {f}));')
    lines.append("return 0;}")
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines))
    exe = tmp_path / "layout"
    subprocess.run([cc, "-std=c99", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)],
                   check=True)
    out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.split("\n")
    got = {(l.split()[0], l.split()[1]): int(l.split()[2]) for l in out if l.strip()}
    for cname, py in structs.items():
        assert got[(cname, "size")] == C.sizeof(py), cname
        for f, _ in py._fields_:
            assert got[(cname, f)] == getattr(py, f).offset, (cname, f)


def test_new_entry_points_validate_on_host():
    """prcr_prefill_capture / prcr_decode_attention / prcr_select_topk reject
    bad arguments before any CUDA call."""
    a = _descs()
    L = prcr.lib()
    st = C.byref(a["st"]); ca = C.byref(a["ca"]); cfg = C.byref(a["cfg"])
    K, V, CO, STAT = FAKE + 2 ** 23, FAKE + 2 ** 24, FAKE + 2 ** 25, FAKE + 2 ** 26
    cap = lambda **k: L.prcr_prefill_capture(cfg, st, ca, k.get("seq", 0), k.get("l0", 0),
                                             k.get("nl", 2), k.get("m0", 0), k.get("mc", 8),
                                             k.get("slot", 0), k.get("k", K), V, 4 * 128, 128,
                                             k.get("coords", CO), k.get("status", STAT), None)
    assert cap(seq=1) == B.EINVAL
    assert cap(l0=1) == B.EINVAL
    assert cap(slot=-1) == B.EINVAL
    assert cap(coords=None) == B.EINVAL
    assert cap(status=None) == B.EINVAL
    assert cap(k=K + 8) == B.EALIGN
    assert cap(mc=0) == B.OK
    # decode: head_dim 64 is allowed, 16 query heads per KV head is not
    Q, QP, SL, OUT = FAKE + 2 ** 27, FAKE + 2 ** 28, FAKE + 2 ** 29, FAKE + 2 ** 30
    dec = lambda **k: L.prcr_decode_attention(cfg, ca, k.get("B", 1), k.get("Hq", 4), Q, QP, SL,
                                              k.get("max_len", 100), k.get("out", OUT), STAT,
                                              None, 0, None)
    assert dec(Hq=3) == B.EINVAL          # not a multiple of the KV heads
    assert dec(Hq=32) == B.EINVAL         # 16 per KV head
    assert dec(max_len=257) == B.EINVAL   # beyond the cache's 256 slots
    assert dec(B=2) == B.EINVAL           # more sequences than the cache holds
    assert dec(out=OUT + 4) == B.EALIGN
    assert dec(B=0) == B.OK
    cfg48 = prcr.rope_cfg(2, 2, 48, (8, 8, 8))
    assert L.prcr_decode_attention(C.byref(cfg48), ca, 1, 4, Q, QP, SL, 10, OUT, STAT, None, 0,
                                   None) == B.EINVAL  # head_dim 48 unsupported by decode
    # select
    IDX, SRO, RTO, WS = FAKE + 2 ** 31, FAKE + 2 ** 32, FAKE + 2 ** 33, FAKE + 2 ** 34
    sel = lambda **k: L.prcr_select_topk(cfg, st, k.get("B", 1), k.get("layer", 0),
                                         k.get("Hq", 4), Q, QP, k.get("k", 8), IDX, SRO, RTO,
                                         None, k.get("ws", WS), k.get("wsb", 1 << 20), None)
    assert sel(k=0) == B.EINVAL
    assert sel(k=65) == B.EINVAL          # more than the 64 store tokens
    assert sel(layer=2) == B.EINVAL
    assert sel(Hq=3) == B.EINVAL
    assert sel(ws=None) == B.EWORKSPACE
    assert sel(wsb=16) == B.EWORKSPACE
    assert prcr.select_workspace_size(2, 4, 64) >= 2 * 4 * 64 * 4 + 2 * 64 * 4


def test_select_cached_validates_on_host():
    """prcr_select_topk_cached rejects bad arguments before any CUDA call:
    the shared selection checks, its own head_dim limit, the image slot
    array and the status word."""
    a = _descs()
    L = prcr.lib()
    ca = C.byref(a["ca"]); cfg = C.byref(a["cfg"])
    Q, QP, IMG, STAT = FAKE + 2 ** 27, FAKE + 2 ** 28, FAKE + 2 ** 29, FAKE + 2 ** 26
    IDX, SRO, RTO, WS = FAKE + 2 ** 31, FAKE + 2 ** 32, FAKE + 2 ** 33, FAKE + 2 ** 34

    def sel(cfg_=cfg, **k):
        return L.prcr_select_topk_cached(cfg_, ca, k.get("B", 1), k.get("layer", 0), k.get("Hq", 4),
                                         k.get("M", 64), k.get("img", IMG), Q, QP, k.get("k", 8),
                                         IDX, SRO, RTO, None, k.get("status", STAT),
                                         k.get("ws", WS), k.get("wsb", 1 << 20), None)
    assert sel(k=0) == B.EINVAL
    assert sel(k=65) == B.EINVAL           # more than the image's 64 tokens
    assert sel(M=0) == B.EINVAL
    assert sel(M=40000) == B.EINVAL        # beyond PRCR_SELECT_MAX_TOKENS
    assert sel(layer=2) == B.EINVAL
    assert sel(Hq=3) == B.EINVAL
    assert sel(B=2) == B.EINVAL            # more sequences than the cache holds
    assert sel(img=None) == B.EINVAL
    assert sel(status=None) == B.EINVAL
    assert sel(img=IMG + 2) == B.EALIGN
    assert sel(ws=None) == B.EWORKSPACE
    assert sel(wsb=16) == B.EWORKSPACE
    assert sel(B=0) == B.OK
    cfg48 = prcr.rope_cfg(2, 2, 48, (8, 8, 8))
    assert sel(cfg_=C.byref(cfg48)) == B.EINVAL  # head_dim 48: the cached path takes 64 and 128
