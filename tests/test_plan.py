"""The attention launch planner, on the CPU: archer_attn_plan_query with an
explicit SM count is host arithmetic (no CUDA call), and the attention calls
launch exactly the plan it returns.  Each expected value is worked out by hand
from the planner's rules, with 128-row query tiles and 128-key tiles:

* T = ceil(P/128) + ceil(G/128) key tiles per item; rows = G (cached step)
  or N (refresh); pairs = ceil(rows/256) * Hq * B two-tile items.
* one tile per CTA when rows <= 128 or 2 * pairs <= SMs;
* with CTAs < SMs and T >= 16, s = min(T, 16, SMs // CTAs) splits of
  per = ceil(T / s) tiles, n_split = ceil(T / per), wanting
  n_split * B * Hq * rows * (4 D + 8) bytes; no split without that workspace;
* two-tile items beyond the SMs: a last wave r = items mod SMs with
  0 < 2 r <= SMs runs as 2 r single-tile CTAs (r extra CTAs);
* persistent (grid = SMs) when the query ranges are whole tile pairs and
  either that tail is empty or items >= 3 SMs; in a cached step the tail then
  runs inside the walk as 2 r single tiles (single_tail = r), in a refresh it
  is walked in pairs (single_tail = 0).
"""
import pytest

from paper_2608_08086_gb300 import build

build.build()                     # the binding refuses to import without the library
from paper_2608_08086_gb300 import archer as A  # noqa: E402

SMS = 152


def plan(B, P, G, Hq, Hkv, D, op=0, ws=0, sms=SMS):
    return A.archer_attn_plan_query(A.make_shape(B, P, G, Hq, Hkv, D), op, ws, sms)


def test_long_prompt_gqa_cached_step_is_persistent():
    # rows 512 -> 2 pairs x 28 heads x 16 = 896 items > 152; 896 mod 152 = 136,
    # 2 * 136 > 152: no tail; ranges whole -> persistent, grid 152; T = 32 + 4
    p = plan(16, 4096, 512, 28, 4, 128)
    assert p == dict(kernel=A.ARCHER_KERNEL_PERSISTENT, tiles_per_cta=2, n_split=1, key_tiles_per_split=36,
                     work_items=896, grid=152, single_tail=0, split_workspace=0)


def test_long_prompt_gqa_refresh_is_persistent_despite_a_small_last_wave():
    # rows 4608 -> 18 pairs x 28 x 16 = 8064 items; 8064 mod 152 = 8 would be a
    # tail, but 8064 >= 3 x 152 -> persistent, and a refresh walks it in pairs
    for op in (A.ARCHER_PLAN_REFRESH_ALL, A.ARCHER_PLAN_REFRESH_FLAGS):
        p = plan(16, 4096, 512, 28, 4, 128, op=op)
        assert (p["kernel"], p["work_items"], p["grid"], p["single_tail"]) == (A.ARCHER_KERNEL_PERSISTENT, 8064, 152, 0)


def test_llada_layer_runs_one_tile_ctas_unsplit():
    # 32 pairs, 2 x 32 <= 152 -> one tile per CTA: 2 x 32 = 64 CTAs; T = 4 + 2 < 16
    p = plan(1, 512, 256, 32, 32, 128, ws=1 << 30)
    assert p == dict(kernel=A.ARCHER_KERNEL_ONE_TILE, tiles_per_cta=1, n_split=1, key_tiles_per_split=6,
                     work_items=64, grid=64, single_tail=0, split_workspace=0)


def test_32_layer_trajectory_is_persistent_with_3_4_items_per_sm():
    # 2 pairs x 32 x 8 = 512 items; 512 mod 152 = 56 (a tail) but 512 >= 456;
    # the walk takes 456 items in pairs, then 112 single tiles on 112 CTAs
    p = plan(8, 1024, 512, 32, 32, 128)
    assert (p["kernel"], p["work_items"], p["grid"], p["key_tiles_per_split"], p["single_tail"]) == (
        A.ARCHER_KERNEL_PERSISTENT, 512, 152, 12, 56)


def test_key_split_needs_its_workspace():
    # 3 pairs x 7 = 21, 2 x 21 <= 152 -> one tile: 3 x 7 = 21 CTAs; T = 13 + 3 = 16;
    # s = min(16, 16, 152 // 21 = 7) = 7, per = 3, n_split = 6;
    # bytes = 6 x 1 x 7 x 384 x (512 + 8) = 8,386,560
    want = 6 * 1 * 7 * 384 * (4 * 128 + 8)
    p = plan(1, 1664, 384, 7, 1, 128, ws=want)
    assert p == dict(kernel=A.ARCHER_KERNEL_ONE_TILE, tiles_per_cta=1, n_split=6, key_tiles_per_split=3,
                     work_items=126, grid=126, single_tail=0, split_workspace=want)
    p = plan(1, 1664, 384, 7, 1, 128, ws=want - 1)
    assert (p["n_split"], p["key_tiles_per_split"], p["grid"], p["split_workspace"]) == (1, 16, 21, want)


def test_split_counts_stay_within_the_key_tiles():
    # D 64, B 2, 70 rows: one tile; CTAs = 1 x 3 x 2 = 6; P 1920: T = 15 + 1 = 16;
    # s = min(16, 16, 25) = 16 -> per 1, n_split 16, 16 x 6 = 96 CTAs
    p = plan(2, 1920, 70, 3, 1, 64, ws=1 << 30)
    assert (p["kernel"], p["n_split"], p["key_tiles_per_split"], p["grid"]) == (A.ARCHER_KERNEL_ONE_TILE, 16, 1, 96)
    assert p["split_workspace"] == 16 * 2 * 3 * 70 * (4 * 64 + 8)
    # P 1930: T = 16 + 1 = 17; s = 16 -> per = 2, n_split = ceil(17 / 2) = 9
    # (none empty), 9 x 6 = 54 CTAs
    p = plan(2, 1930, 70, 3, 1, 64, ws=1 << 30)
    assert (p["n_split"], p["key_tiles_per_split"], p["grid"]) == (9, 2, 54)
    # P 1792: T = 14 + 1 = 15 < 16: no split however idle the SMs
    p = plan(2, 1792, 70, 3, 1, 64, ws=1 << 30)
    assert (p["n_split"], p["grid"], p["split_workspace"]) == (1, 6, 0)


def test_two_tile_grid_with_a_single_tile_tail():
    # 1 pair x 32 x 5 = 160 items > 152; r = 8, 2 x 8 <= 152 -> tail 8;
    # 160 < 456 -> not persistent: 152 pair CTAs + 2 x 8 single-tile CTAs = 168
    p = plan(5, 512, 256, 32, 32, 128)
    assert p == dict(kernel=A.ARCHER_KERNEL_TWO_TILE, tiles_per_cta=2, n_split=1, key_tiles_per_split=6,
                     work_items=160, grid=168, single_tail=8, split_workspace=0)


def test_two_tile_grid_within_one_wave():
    # 96 pairs: 2 x 96 > 152 -> two tiles; 96 <= 152 -> neither tail nor persistent
    p = plan(3, 512, 256, 32, 32, 128)
    assert (p["kernel"], p["grid"], p["single_tail"]) == (A.ARCHER_KERNEL_TWO_TILE, 96, 0)


def test_partial_tile_pairs_are_not_persistent():
    # refresh with flags, P 100: rows 356 -> 2 pairs x 28 x 16 = 896 items, no
    # tail (896 mod 152 = 136); a refreshed range of 356 rows is not whole pairs
    p = plan(16, 100, 256, 28, 4, 128, op=A.ARCHER_PLAN_REFRESH_FLAGS)
    assert (p["kernel"], p["grid"], p["work_items"]) == (A.ARCHER_KERNEL_TWO_TILE, 896, 896)
    # the cached step of the same shape (256 rows) is whole pairs: persistent
    p = plan(16, 100, 256, 28, 4, 128)
    assert (p["kernel"], p["grid"], p["work_items"]) == (A.ARCHER_KERNEL_PERSISTENT, 152, 448)


def test_plan_follows_the_sm_count():
    # the same launch on a GPU of 1024 SMs: 896 items fit in one wave
    p = plan(16, 4096, 512, 28, 4, 128, sms=1024)
    assert (p["kernel"], p["grid"]) == (A.ARCHER_KERNEL_TWO_TILE, 896)


def test_batch_zero_and_bad_arguments():
    assert plan(0, 512, 256, 32, 32, 128)["grid"] == 0
    with pytest.raises(A.ArcherError):
        A.archer_attn_plan_query(A.make_shape(1, 512, 256, 32, 32, 128), 7, 0, SMS)
    with pytest.raises(A.ArcherError):
        plan(1, 512, 256, 32, 32, 96)                       # head_dim 96
    with pytest.raises(A.ArcherError):
        plan(1, 512, 256, 30, 4, 128)                       # 30 % 4 != 0
