"""Host logic of bench.py that needs no GPU: the code digest that decides
whether the committed DRAM traffic still describes the kernels."""
import os
import shutil

import bench

CSRC = os.path.join(bench.ROOT, "paper_2608_17310_gb300", "csrc")


def test_strip_comments_keeps_literals_and_drops_comments():
    src = 'a = "x // y /* z */"; // gone\n/* gone\n too */ b = \'/\';  \n\n  c  =  1;\n'
    assert bench.strip_comments(src) == 'a = "x // y /* z */";\nb = \'/\';\nc = 1;'
    assert bench.strip_comments('asm("mov.b32 %0, %1;" : "=r"(x));') == \
        'asm("mov.b32 %0, %1;" : "=r"(x));'


def _copy_sources(tmp_path):
    for f in bench.KERNEL_SOURCES:
        shutil.copy(os.path.join(CSRC, f), tmp_path / f)
    return str(tmp_path)


def test_comment_edit_keeps_the_digest_and_code_edit_changes_it(tmp_path):
    d = _copy_sources(tmp_path)
    base = bench.kernel_code_digest(d)
    assert base == bench.kernel_code_digest(CSRC)
    p = tmp_path / "es_noise.cuh"
    text = p.read_text()
    p.write_text("// a new comment line\n" + text.replace("\n", "   \n", 3) + "\n/* tail */\n")
    assert bench.kernel_code_digest(d) == base
    p.write_text(text.replace("0xD2511F53u", "0xD2511F55u"))
    assert bench.kernel_code_digest(d) != base


def test_traffic_file_is_keyed_by_a_well_formed_digest():
    rows = [line.split() for line in open(os.path.join(bench.ROOT, "profiles", "dram_traffic.txt"))
            if line.strip() and not line.startswith("#")]
    assert {r[0] for r in rows} == {"restore_perturb", "restore", "update_perturb", "update"}
    for kind, per_param, digest in rows:
        assert 2.0 < float(per_param) < 8.0
        assert len(digest) == 16 and int(digest, 16) >= 0


def test_pipe_occupancy_file_is_keyed_by_the_current_code():
    occ = bench.pipe_occupancy("restore_perturb")
    rows = [line.split() for line in open(os.path.join(bench.ROOT, "profiles", "pipe_occupancy.txt"))
            if line.strip() and not line.startswith("#")]
    assert {r[0] for r in rows} == {"restore_perturb", "restore", "update_perturb", "update"}
    if all(r[3] == bench.kernel_code_digest() for r in rows):
        # the two pipes overlap, so their sum may exceed 100 %
        assert occ is not None and 90.0 < occ["sum_pct"] < 200.0
        for r in rows:
            assert 0.0 < float(r[1]) <= 100.0 and 0.0 < float(r[2]) <= 100.0
    assert bench.pipe_occupancy("perturb") is None


def test_hugepage_fraction_of_an_anonymous_mapping_is_a_fraction():
    import ctypes
    import mmap
    import numpy as np
    buf = bench.PinnedHostBuffer.__new__(bench.PinnedHostBuffer)
    buf.nbytes = 16 << 20
    m = mmap.mmap(-1, buf.nbytes, flags=mmap.MAP_PRIVATE | mmap.MAP_ANONYMOUS)
    buf.addr = ctypes.addressof(ctypes.c_char.from_buffer(m))
    np.frombuffer(m, dtype=np.uint8)[::4096] = 1
    frac = buf.hugepage_fraction()
    assert frac is None or 0.0 <= frac <= 1.0
    buf.addr = None
    assert buf.hugepage_fraction() is None


def test_copy_groups_cover_every_tensor_with_a_shrinking_tail():
    from paper_2608_17310_gb300 import inputs as I
    for name in ("qwen27b", "qwen4b", "qwen4b_4layer", "toy"):
        sizes = [s.numel for s in I.shapes_for(name)]
        total = sum(sizes)
        ends = bench.copy_groups(sizes, 8)
        starts = [0] + ends[:-1]
        assert ends[-1] == len(sizes) and len(ends) <= 12
        assert all(b > a for a, b in zip(starts, ends))   # non-empty, in order
        group = [sum(sizes[a:b]) for a, b in zip(starts, ends)]
        # the last group: at most 1/32 of the elements, or a single tensor
        assert ends[-1] - starts[-1] == 1 or group[-1] <= total / 32
    # on the 27B-shaped set the groups shrink towards the end: each of the
    # last three at most half the one before it (within one tensor)
    sizes = [s.numel for s in I.shapes_for("qwen27b")]
    ends = bench.copy_groups(sizes, 8)
    starts = [0] + ends[:-1]
    group = [sum(sizes[a:b]) for a, b in zip(starts, ends)]
    big = max(sizes)
    assert group[-1] <= group[-2] and group[-2] <= group[-3] / 2 + big
    assert bench.copy_groups([5], 8) == [1]
    assert bench.copy_groups([1] * 64, 8)[-1] == 64
