"""CPU tests of the C ABI: the library builds and loads, exports every entry
point include/moara.h declares, and its host-only functions (memory model,
rank table, workspace sizes, hyper-parameter defaults, status strings) are
right.  No compute call is made here."""

import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "moara.h")
GOLDEN = os.path.join(ROOT, "tests", "golden")


@pytest.fixture(scope="module")
def M():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2609_15037_gb300 as pkg
    return pkg


def _declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(moara_[a-z_0-9]+)\s*\(", src)))


def test_exports_every_declared_symbol(M):
    lib = ctypes.CDLL(M.binding.LIB_PATH)
    names = _declared()
    assert len(names) >= 15
    for name in names:
        assert hasattr(lib, name), name
    assert sorted(M.binding.EXPORTED) == names


def test_default_hparams_follow_paper(M):
    hp = M.moara_default_hparams()
    assert hp.beta1 == pytest.approx(0.9) and hp.beta2 == pytest.approx(0.999)
    assert hp.adam_eps == pytest.approx(1e-6) and hp.decomp_eps == pytest.approx(1e-12)
    assert hp.scale == pytest.approx(0.25) and hp.refresh_interval == 200
    assert hp.decompose == 1 and hp.refresh_src == M.MOARA_REFRESH_SRC_V
    assert hp.clip_norm == 0.0           # clipping off unless asked for (App. D.2: 7B runs only)


def test_hparams_struct_matches_header(M):
    """The binding's struct has the C layout: the library's defaults land in
    the right fields, including the last one."""
    hp = M.moara_default_hparams()
    assert hp.block_size == 128 and hp.power_iters == 4 and hp.oversample == 32 and hp.ritz_iters == 3
    assert ctypes.sizeof(M.binding.moara_hparams) == 80
    assert hp.proj_rule == M.MOARA_PROJ_LEFT and hp.state_dtype == M.MOARA_DTYPE_F32


def test_flatten_shape_through_the_abi(M):
    """App. B flatten rule via moara_flatten_shape, against the oracle's."""
    from oracle import moara_ref as o
    for shape in [(8, 3, 3, 3), (4096, 11008), (5,), (2, 3, 4, 5, 6)]:
        assert M.moara_flatten_shape(shape) == o.flatten_shape(shape)
    with pytest.raises(M.MoaraError) as ei:
        M.moara_flatten_shape((3, 0))
    assert ei.value.code == M.MOARA_ERR_INVALID_ARG
    with pytest.raises(M.MoaraError) as ei:
        M.moara_flatten_shape((2, 1 << 20, 1 << 12))
    assert ei.value.code == M.MOARA_ERR_SHAPE


def _golden(name):
    rows = {}
    for line in open(os.path.join(GOLDEN, name)):
        if line.strip() and not line.startswith("#"):
            p = line.split()
            rows[p[0]] = p[1:]
    return rows


@pytest.mark.parametrize("model", ["350M", "1B", "7B"])
def test_state_bytes_reproduce_printed_memory_table(M, model):
    """moara_state_bytes summed over the target matrices plus the model's
    other parameters (untied 32000-token embedding and head with 2-byte Adam
    states, fp32 norms) gives the printed optimizer-state MiB values."""
    row = _golden("memory_table.txt")[model]
    h, f, L, B, rb = (int(x) for x in row[:5])
    printed = [float(x) for x in row[5:]]
    shp = [(h, h), (h, h), (h, h), (h, h), (f, h), (f, h), (h, f)]
    aware = M.moara_rank_table(rb, 0b11, 1 << 6, rb // 2)
    other = 2 * 32000 * h * 2 * 2 + (2 * L + 1) * h * 4

    def total(ranks, dec):
        return L * sum(M.moara_state_bytes(m, n, ranks[i], B, 2, 4, M.MOARA_DRULE_MAX, dec)
                       for i, (m, n) in enumerate(shp)) + other

    got = [total([rb] * 7, 0), total([rb] * 7, 1), total(aware, 0), total(aware, 1)]
    for g, p in zip(got, printed):
        assert round(g / 2 ** 20, 2) == pytest.approx(p, abs=1e-9)


def test_state_bytes_left_projector_rule(M):
    assert M.moara_state_bytes(100, 300, 10, 64, 4, 4, M.MOARA_DRULE_N, 1) == \
        2 * 4 * 10 * 300 + 2 * 4 * 100 * 5
    assert M.moara_state_bytes(100, 300, 10, 64, 4, 4, M.MOARA_DRULE_N, 0) == 2 * 4 * 10 * 300


def test_rank_table_final_allocation_and_budget(M):
    ours = [int(x) for x in _golden("rank_allocations.txt")["Ours"]]
    assert M.moara_rank_table(256, 0b11, 1 << 6, 128) == ours
    for rb in (256, 512, 1024):
        t = M.moara_rank_table(rb, 0b11, 1 << 6, rb // 2)
        assert t == [rb // 2, rb // 2, rb, rb, rb, rb, 2 * rb] and sum(t) == 7 * rb
    t = M.moara_rank_table(512, 0b111, (1 << 5) | (1 << 6), 101)
    assert sum(t) == 7 * 512 and t[5] == 512 + 152 and t[6] == 512 + 151


def test_rank_table_rejects_bad_input(M):
    with pytest.raises(M.binding.MoaraError):
        M.moara_rank_table(256, 0b1, 0b1, 10)          # overlap
    with pytest.raises(M.binding.MoaraError):
        M.moara_rank_table(256, 0b1, 0, 10)            # donors, no receivers
    with pytest.raises(M.binding.MoaraError):
        M.moara_rank_table(256, 0b1, 0b10, 256)        # delta_r >= r_base
    with pytest.raises(M.binding.MoaraError):
        M.moara_rank_table(256, 1 << 7, 0b10, 1)       # unknown module bit


def test_state_and_workspace_validation(M):
    with pytest.raises(M.binding.MoaraError) as e:
        M.moara_state_bytes(10, 10, 11, 4, 4, 4)
    assert e.value.code == M.MOARA_ERR_RANK
    with pytest.raises(M.binding.MoaraError) as e:
        M.moara_workspace_bytes(10, 10, 2, 0)
    assert e.value.code == M.MOARA_ERR_SHAPE
    ws = M.moara_workspace_bytes(4096, 11008, 2048, 128)
    assert ws >= 4 * 2048 * 11008 + 8 * 4096 * 86
    assert ws % 256 == 0


def test_status_strings(M):
    assert M.moara_status_string(0) == "ok"
    assert "timed out" in M.moara_status_string(M.MOARA_ERR_DEVICE_TIMEOUT)
    assert M.moara_status_string(12345) == "unknown status"


def test_create_without_gpu_fails_cleanly(M):
    torch = pytest.importorskip("torch")
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    with pytest.raises(M.binding.MoaraError) as e:
        M.moara_create(M.moara_default_hparams(), 0)
    assert e.value.code == M.MOARA_ERR_CUDA
    hp = M.moara_default_hparams()
    hp.block_size = 0
    with pytest.raises(M.binding.MoaraError) as e:
        M.moara_create(hp, 0)
    assert e.value.code == M.MOARA_ERR_SHAPE
