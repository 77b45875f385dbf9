"""C-ABI checks that need no GPU: the library loads, exports every symbol that
include/rc.h declares, validates ops, and canonicalises schedules."""
import ctypes
import os
import re

import pytest

from paper_2506_01374_gb300 import rc

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared_functions():
    names = set()
    for h in os.listdir(os.path.join(ROOT, "include")):
        if not h.endswith(".h"):
            continue
        src = open(os.path.join(ROOT, "include", h)).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        for m in re.finditer(r"^\s*(?:const\s+)?[A-Za-z_][\w\s\*]*?\b(rc_\w+)\s*\(", src, flags=re.M):
            names.add(m.group(1))
    return names


def test_library_exports_every_declared_symbol():
    names = _declared_functions()
    assert {"rc_op_describe", "rc_schedule_apply", "rc_candidate_measure", "rc_search_step"} <= names
    L = ctypes.CDLL(rc.LIB_PATH)
    missing = [n for n in sorted(names) if not hasattr(L, n)]
    assert not missing, missing


def test_op_validation_errors():
    with pytest.raises(rc.RcError) as e:
        rc.Op(rc.OP_GEMM_F32, m=0, n=4, k=4)
    assert e.value.status == rc.ERR_INVALID_ARG
    with pytest.raises(rc.RcError) as e:
        rc.Op(rc.OP_ATTENTION, batch=1, seq=16, heads_q=4, heads_kv=2, head_dim=64)
    assert e.value.status == rc.ERR_UNSUPPORTED_OP
    with pytest.raises(rc.RcError) as e:
        rc.Op(rc.OP_ATTENTION, batch=1, seq=16, heads_q=3, heads_kv=2, head_dim=128)
    assert e.value.status == rc.ERR_INVALID_ARG
    with pytest.raises(rc.RcError) as e:
        rc.Op(99)
    assert e.value.status == rc.ERR_UNSUPPORTED_OP


def test_algorithmic_work_of_the_workloads():
    # Flop counts of the five workloads (2 flops per multiply-add).
    assert rc.Op(rc.OP_GEMM_F32, m=256, n=256, k=256).info["flops"] == 2 * 256 ** 3
    mlp = rc.Op(rc.OP_MLP, m=2048, n=14336, k=4096).info
    assert mlp["flops"] == 6 * 2048 * 14336 * 4096 and mlp["bound"] == "tensor"
    att = rc.Op(rc.OP_ATTENTION, batch=1, seq=2048, heads_q=32, heads_kv=8, head_dim=128, causal=1).info
    assert att["flops"] == 4 * 128 * 32 * 2048 * 2049 // 2
    conv = rc.Op(rc.OP_CONV2D, img_n=2, img_h=64, img_w=64, c_in=320, c_out=320, kr=3, ks=3, stride=1, pad=1,
                 flags=rc.EPI_BIAS | rc.EPI_SILU).info
    assert conv["flops"] == 2 * 8192 * 320 * 2880
    moe = rc.Op(rc.OP_MOE, tokens=4096, hidden=7168, experts=64, inter=2048, top_k=8).info
    assert moe["flops"] == 6 * 4096 * 8 * 7168 * 2048


def test_schedule_canonical_form_last_writer_wins():
    op = rc.Op(rc.OP_GEMM_F32, m=256, n=256, k=256, flags=rc.EPI_BIAS | rc.EPI_RELU)
    a = op.schedule(rc.T(rc.T_TILE_SIZE, 32, axis=0), rc.T(rc.T_TILE_SIZE, 64, axis=0), rc.T(rc.T_UNROLL, 4))
    b = op.schedule(rc.T(rc.T_UNROLL, 4), rc.T(rc.T_TILE_SIZE, 64, axis=0))
    assert a.hash == b.hash and str(a) == str(b)
    assert a.knobs()["tile_m"] == 64 and a.knobs()["unroll"] == 4
    c = op.schedule(rc.T(rc.T_TILE_SIZE, 32, axis=1), base=a)
    assert c.knobs()["tile_n"] == 32 and c.knobs()["tile_m"] == 64 and c.hash != a.hash
    p0 = op.schedule()
    assert (p0.knobs()["tile_m"], p0.knobs()["tile_n"], p0.knobs()["tile_k"], p0.knobs()["unroll"]) == (16, 16, 16, 1)


def test_gemm_f32_space_is_the_54_point_grid():
    op = rc.Op(rc.OP_GEMM_F32, m=256, n=256, k=256)
    space = op.transform_space()
    got = [(t.kind, t.axis, t.value[0]) for t in space]
    want = [(rc.T_TILE_SIZE, ax, v) for ax in range(3) for v in (16, 32, 64)] + [(rc.T_UNROLL, 0, 1),
                                                                                (rc.T_UNROLL, 0, 4)]
    assert got == want
    hashes = set()
    for bm in (16, 32, 64):
        for bn in (16, 32, 64):
            for bk in (16, 32, 64):
                for u in (1, 4):
                    s = op.schedule(rc.T(rc.T_TILE_SIZE, bm, axis=0), rc.T(rc.T_TILE_SIZE, bn, axis=1),
                                    rc.T(rc.T_TILE_SIZE, bk, axis=2), rc.T(rc.T_UNROLL, u))
                    hashes.add(s.hash)
    assert len(hashes) == 54


def test_illegal_schedules_are_rejected():
    op = rc.Op(rc.OP_LINEAR, m=512, n=1024, k=1024)
    for t in [rc.T(rc.T_TILE_SIZE, 96, axis=1), rc.T(rc.T_SPLIT_K, 3), rc.T(rc.T_UNROLL, 2),
              rc.T(rc.T_TILE_SIZE, 64, axis=5), rc.T(rc.T_PIPELINE_STAGES, 2, stage=1)]:
        with pytest.raises(rc.RcError) as e:
            op.schedule(t)
        assert e.value.status == rc.ERR_ILLEGAL_SCHEDULE
    # 256-wide tiles with 6 stages overflow 227 KB of shared memory
    with pytest.raises(rc.RcError) as e:
        op.schedule(rc.T(rc.T_TILE_SIZE, 256, axis=1), rc.T(rc.T_PIPELINE_STAGES, 6))
    assert e.value.status == rc.ERR_ILLEGAL_SCHEDULE
    ok = op.schedule(rc.T(rc.T_TILE_SIZE, 256, axis=1), rc.T(rc.T_PIPELINE_STAGES, 4))
    assert ok.knobs()["tile_n"] == 256


def test_composite_op_stages_are_independent():
    op = rc.Op(rc.OP_MLP, m=256, n=512, k=256)
    s = op.schedule(rc.T(rc.T_TILE_SIZE, 128, axis=1, stage=0), rc.T(rc.T_TILE_SIZE, 256, axis=1, stage=1),
                    rc.T(rc.T_SPLIT_K, 2, stage=1), rc.T(rc.T_FUSE, 1, stage=0))
    assert s.num_stages == 2
    assert s.knobs(0)["tile_n"] == 128 and s.knobs(0)["fuse"] == 1
    assert s.knobs(1)["tile_n"] == 256 and s.knobs(1)["split_k"] == 2
    with pytest.raises(rc.RcError):
        op.schedule(rc.T(rc.T_SPLIT_K, 2, stage=0))  # split-K belongs to the down GEMM


def test_schedule_string_round_trip_size():
    op = rc.Op(rc.OP_MOE, tokens=64, hidden=128, experts=8, inter=64, top_k=2)
    s = op.schedule()
    txt = str(s)
    assert txt.startswith("op=moe;s0:") and ";s2:" in txt


def _decoder(**kw):
    a = dict(tokens=2048, hidden=4096, inter=14336, heads_q=32, heads_kv=8, head_dim=128)
    a.update(kw)
    return rc.Op(rc.OP_DECODER_LAYER, **a)


def test_decoder_layer_op_work_and_validation():
    info = _decoder().info
    T, H, I, hq, hkv = 2048, 4096, 14336, 32 * 128, 8 * 128
    want = 2 * T * H * (hq + 2 * hkv) + 4 * 128 * 32 * T * (T + 1) // 2 + 2 * T * hq * H + 6 * T * H * I
    assert info["flops"] == want and info["bound"] == "tensor" and info["n_tensors"] == 8
    for kw, st in [(dict(hidden=4000), rc.ERR_UNSUPPORTED_OP), (dict(head_dim=64), rc.ERR_UNSUPPORTED_OP),
                   (dict(heads_q=12, heads_kv=8), rc.ERR_INVALID_ARG), (dict(tokens=0), rc.ERR_INVALID_ARG),
                   (dict(inter=100), rc.ERR_UNSUPPORTED_OP), (dict(norm_eps=-1.0), rc.ERR_INVALID_ARG)]:
        with pytest.raises(rc.RcError) as e:
            _decoder(**kw)
        assert e.value.status == st, kw
    # head_dim 0 takes the default of 128
    assert _decoder(head_dim=0).info["flops"] == want


def test_decoder_layer_schedule_has_six_independent_stages():
    op = _decoder(tokens=256, hidden=512, inter=768, heads_q=4, heads_kv=2)
    p0 = op.schedule()
    assert p0.num_stages == 6 and str(p0).startswith("op=decoder_layer;s0:") and ";s5:" in str(p0)
    s = op.schedule(rc.T(rc.T_TILE_SIZE, 4, axis=0, stage=1), rc.T(rc.T_FUSE, 1, stage=4),
                    rc.T(rc.T_TILE_SIZE, 128, axis=1, stage=2), rc.T(rc.T_TILE_SIZE, 256, axis=0, stage=5))
    assert s.knobs(1)["tile_m"] == 4 and s.knobs(4)["fuse"] == 1
    assert s.knobs(2)["tile_n"] == 128 and s.knobs(5)["tile_m"] == 256 and s.knobs(0) == p0.knobs(0)
    stages = {t.stage for t in op.transform_space()}
    assert stages == set(range(6))
    for t in [rc.T(rc.T_TILE_SIZE, 3, axis=0, stage=1),       # tokens per CTA outside {1, 2, 4, 8}
              rc.T(rc.T_SPLIT_K, 2, stage=5),                 # no split-K in the layer's GEMMs
              rc.T(rc.T_FUSE, 1, stage=0),                    # fusion belongs to the gate/up GEMM
              rc.T(rc.T_LOOP_ORDER, 2, stage=2),              # persistent attention needs its own knobs
              rc.T(rc.T_TILE_SIZE, 64, axis=1, stage=6)]:     # no seventh stage
        with pytest.raises(rc.RcError) as e:
            op.schedule(t)
        assert e.value.status == rc.ERR_ILLEGAL_SCHEDULE, t
    # P0's workspace: a, qkv, Q, K, V, o, h1, b, the SwiGLU output, gate|up (unfused) and V transposed
    T, H, I, hq, hkv = 256, 512, 768, 512, 256
    want = 2 * (T * H + T * (hq + 2 * hkv) + T * hq + 2 * T * hkv + T * hq + 2 * T * H + T * I + 2 * T * I + hkv * T)
    assert op.info["workspace_bytes"] == want


def test_binding_constants_match_the_header():
    src = re.sub(r"/\*.*?\*/", "", open(os.path.join(ROOT, "include", "rc.h")).read(), flags=re.S)
    assert int(re.search(r"#define RC_MAX_STAGES (\d+)", src).group(1)) == rc.MAX_STAGES
    kinds = re.search(r"typedef enum \{([^{}]*)\} rc_op_kind;", src).group(1)
    assert int(re.search(r"RC_OP_DECODER_LAYER = (\d+)", kinds).group(1)) == rc.OP_DECODER_LAYER
    # the search options end with the task fields (stage_mask, root) in that order
    opts = re.search(r"typedef struct \{([^{}]*)\} rc_search_opts;", src).group(1)
    names = re.findall(r"(\w+);", opts)
    assert names == [f for f, _ in rc.SearchOpts._fields_]


def test_vectorize_offered_and_normalised_where_no_pass_runs():
    # Vectorize sets the access width of a stage's memory-bound pass; a stage that runs none keeps the default
    op = rc.Op(rc.OP_MLP, m=64, n=128, k=64)
    kinds = {(t.kind, t.stage) for t in op.transform_space()}
    assert (rc.T_VECTORIZE, 0) in kinds and (rc.T_VECTORIZE, 1) in kinds
    fused = op.schedule(rc.T(rc.T_FUSE, 1, stage=0), rc.T(rc.T_VECTORIZE, 4, stage=0))
    assert fused.knobs(0)["vec"] == 16 and str(fused) == str(op.schedule(rc.T(rc.T_FUSE, 1, stage=0)))
    unfused = op.schedule(rc.T(rc.T_VECTORIZE, 8, stage=0))
    assert unfused.knobs(0)["vec"] == 8 and str(unfused) != str(op.schedule())
    no_split = op.schedule(rc.T(rc.T_VECTORIZE, 4, stage=1))
    assert no_split.knobs(1)["vec"] == 16
    split = op.schedule(rc.T(rc.T_SPLIT_K, 2, stage=1), rc.T(rc.T_VECTORIZE, 4, stage=1))
    assert split.knobs(1)["vec"] == 4
    with pytest.raises(rc.RcError) as e:
        op.schedule(rc.T(rc.T_VECTORIZE, 2, stage=0))
    assert e.value.status == rc.ERR_ILLEGAL_SCHEDULE
    moe = rc.Op(rc.OP_MOE, tokens=64, hidden=128, experts=4, inter=64, top_k=2)
    g = moe.schedule(rc.T(rc.T_VECTORIZE, 4, stage=0))
    assert g.knobs(0)["vec"] == 4
    # rows gathered inside the gate/up GEMM: stage 0 runs no gather pass
    assert moe.schedule(rc.T(rc.T_COMPUTE_LOCATION, 1, stage=1), rc.T(rc.T_VECTORIZE, 4, stage=0)).knobs(0)["vec"] == 16
    att = rc.Op(rc.OP_ATTENTION, batch=1, seq=128, heads_q=2, heads_kv=1, head_dim=128, causal=1)
    assert all(t.kind != rc.T_VECTORIZE for t in att.transform_space())


def test_two_query_tile_attention_canonical_form_and_legality():
    op = rc.Op(rc.OP_ATTENTION, batch=1, seq=2048, heads_q=32, heads_kv=8, head_dim=128, causal=1)
    # TileSize M = 256 selects the two-query-tile kernel whatever the other families' knobs say
    s = op.schedule(rc.T(rc.T_TILE_SIZE, 64, axis=1), rc.T(rc.T_PARALLEL, 2), rc.T(rc.T_UNROLL, 2),
                    rc.T(rc.T_COMPUTE_LOCATION, 0), rc.T(rc.T_TILE_SIZE, 256, axis=0))
    k = s.knobs(0)
    assert (k["tile_m"], k["tile_n"], k["persistent"], k["location"], k["unroll"]) == (256, 128, 1, 1, 1)
    assert str(s) == str(op.schedule(rc.T(rc.T_TILE_SIZE, 256, axis=0), rc.T(rc.T_PARALLEL, 1)))
    # two 32 KB query tiles, a 128-key K ring and a two-slot V ring: at most three K stages fit 227 KB
    for st in (1, 2, 3):
        op.schedule(rc.T(rc.T_TILE_SIZE, 256, axis=0), rc.T(rc.T_PIPELINE_STAGES, st))
    with pytest.raises(rc.RcError):
        op.schedule(rc.T(rc.T_TILE_SIZE, 256, axis=0), rc.T(rc.T_PIPELINE_STAGES, 4))
    # the transposed V needs 16-byte rows: seq % 8 == 0
    odd = rc.Op(rc.OP_ATTENTION, batch=1, seq=300, heads_q=4, heads_kv=2, head_dim=128, causal=1)
    with pytest.raises(rc.RcError):
        odd.schedule(rc.T(rc.T_TILE_SIZE, 256, axis=0), rc.T(rc.T_LAYOUT, 1))
    assert any(t.kind == rc.T_TILE_SIZE and t.axis == 0 and t.value[0] == 256 for t in op.transform_space())


def test_persistent_pairs_take_256_column_tiles():
    # two 256-column accumulators fill a pair's 512 TMEM columns: legal (the launcher keeps one CTA per SM)
    op = rc.Op(rc.OP_LINEAR, m=2048, n=4096, k=14336)
    for tn in (224, 256):
        s = op.schedule(rc.T(rc.T_TILE_SIZE, 256, axis=0), rc.T(rc.T_TILE_SIZE, tn, axis=1), rc.T(rc.T_PARALLEL, 1))
        assert s.knobs(0)["persistent"] == 1 and s.knobs(0)["tile_n"] == tn
    mlp = rc.Op(rc.OP_MLP, m=2048, n=14336, k=4096)
    s = mlp.schedule(rc.T(rc.T_TILE_SIZE, 256, axis=0, stage=0), rc.T(rc.T_TILE_SIZE, 128, axis=1, stage=0),
                     rc.T(rc.T_TILE_SIZE, 128, axis=2, stage=0), rc.T(rc.T_PIPELINE_STAGES, 3, stage=0),
                     rc.T(rc.T_PARALLEL, 1, stage=0), rc.T(rc.T_FUSE, 1, stage=0))
    assert s.knobs(0)["persistent"] == 1 and s.knobs(0)["tile_k"] == 128


def test_moe_split_segments_canonical_form():
    op = rc.Op(rc.OP_MOE, tokens=4096, hidden=7168, experts=64, inter=2048, top_k=8)
    both = op.schedule(rc.T(rc.T_TILE_SIZE, 256, axis=0, stage=1), rc.T(rc.T_LAYOUT, 1, stage=1),
                       rc.T(rc.T_TILE_SIZE, 256, axis=0, stage=2), rc.T(rc.T_LAYOUT, 1, stage=2))
    assert both.knobs(1)["layout"] == 1 and both.knobs(2)["layout"] == 1
    # single-CTA M tiles have no remainder to split off: the canonical form drops the layout
    single = op.schedule(rc.T(rc.T_LAYOUT, 1, stage=1), rc.T(rc.T_TILE_SIZE, 128, axis=0, stage=1))
    assert single.knobs(1)["layout"] == 0
    assert str(single) == str(op.schedule(rc.T(rc.T_TILE_SIZE, 128, axis=0, stage=1)))
    # the in-GEMM row gather needs one CTA per tile, so it leaves nothing to split either
    g = op.schedule(rc.T(rc.T_TILE_SIZE, 256, axis=0, stage=1), rc.T(rc.T_LAYOUT, 1, stage=1),
                    rc.T(rc.T_TILE_SIZE, 128, axis=0, stage=1), rc.T(rc.T_COMPUTE_LOCATION, 1, stage=1))
    assert g.knobs(1)["layout"] == 0 and g.knobs(1)["location"] == 1


def test_moe_exchanged_operands_canonical_form_and_legality():
    # Layout 2 of the grouped GEMMs: weights on UMMA M, each expert's tokens on N (token tiles of 64,
    # 128 or 256 rows: 2x the SwiGLU output tile in stage 1, the N tile in stage 2), one CTA or a pair
    op = rc.Op(rc.OP_MOE, tokens=4096, hidden=7168, experts=64, inter=2048, top_k=8)
    T = rc.T
    s = op.schedule(T(rc.T_LAYOUT, 2, stage=1), T(rc.T_TILE_SIZE, 128, axis=1, stage=1),
                    T(rc.T_LAYOUT, 2, stage=2), T(rc.T_TILE_SIZE, 256, axis=1, stage=2), T(rc.T_PARALLEL, 1, stage=2))
    assert s.knobs(1)["layout"] == 2 and s.knobs(2)["layout"] == 2 and s.knobs(2)["persistent"] == 1
    # unlike layout 1, layout 2 stays on single-CTA tiles, and on CTA pairs
    assert op.schedule(T(rc.T_LAYOUT, 2, stage=1)).knobs(1)["layout"] == 2
    pair = op.schedule(T(rc.T_LAYOUT, 2, stage=2), T(rc.T_TILE_SIZE, 256, axis=0, stage=2),
                       T(rc.T_TILE_SIZE, 256, axis=1, stage=2), T(rc.T_PIPELINE_STAGES, 4, stage=2))
    assert pair.knobs(2)["layout"] == 2 and pair.knobs(2)["tile_m"] == 256
    assert str(pair) != str(op.schedule(T(rc.T_TILE_SIZE, 256, axis=0, stage=2), T(rc.T_TILE_SIZE, 256, axis=1, stage=2),
                                        T(rc.T_PIPELINE_STAGES, 4, stage=2)))
    illegal = [
        [T(rc.T_LAYOUT, 2, stage=2), T(rc.T_TILE_SIZE, 224, axis=1, stage=2)],  # token tile of 224 rows
        [T(rc.T_LAYOUT, 2, stage=2), T(rc.T_FUSE, 1, stage=2)],  # the atomic combine epilogue
        [T(rc.T_LAYOUT, 2, stage=1), T(rc.T_COMPUTE_LOCATION, 1, stage=1)],  # rows gathered in the GEMM
        # a single-CTA ring of 4 stages of 256 token rows and two 128-row weight boxes, K 128: 512 KB
        [T(rc.T_LAYOUT, 2, stage=1), T(rc.T_TILE_SIZE, 128, axis=1, stage=1), T(rc.T_TILE_SIZE, 128, axis=2, stage=1),
         T(rc.T_PIPELINE_STAGES, 4, stage=1)],
    ]
    for ts in illegal:
        with pytest.raises(rc.RcError):
            op.schedule(*ts)
    # the search's space offers the layout on both grouped GEMMs
    kinds = {(t.kind, t.stage, t.value[0]) for t in op.transform_space()}
    assert (rc.T_LAYOUT, 1, 2) in kinds and (rc.T_LAYOUT, 2, 2) in kinds
