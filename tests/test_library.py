"""The C-ABI library builds, loads and exports every function include/dvi.h
declares; host-side validation rejects bad configurations without a GPU."""
import ctypes
import os
import re

import pytest

from paper_2510_05421_gb300 import build as build_mod
from paper_2510_05421_gb300 import dvi as D
from workloads import WORKLOADS, tiny_shape

HEADER = os.path.join(os.path.dirname(os.path.dirname(__file__)), "include", "dvi.h")


@pytest.fixture(scope="module")
def L():
    if not os.path.exists(D.LIB_PATH):
        build_mod.build()
    return D.lib()


def declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(dvi_[a-z_]+)\s*\(", src)))


def test_exports_every_declared_function(L):
    names = declared()
    assert len(names) >= 12
    for n in names:
        assert hasattr(L, n), n
    assert sorted(D.EXPORTS) == names


def _cfgs(w, **rt):
    s = w.shape
    cfg = D.ModelConfig(s.n_layers, s.d_model, s.n_heads, s.n_kv_heads, s.head_dim, s.d_ffn, s.vocab, w.split_k,
                        w.lora_rank, 1.0, s.rms_eps, s.rope_theta, D.DVI_BF16 if w.dtype == "bf16" else D.DVI_F32)
    base = dict(batch=w.batch, k_spec=w.k_spec, max_seq_len=w.prompt_len[1] + w.gen_tokens + 64,
                log_steps=w.update_every, head_mode=0, max_prefill_chunk=128, use_graphs=1, bonus=0,
                persistent=0, chain_counters=0, megakernel=0)
    base.update(rt)
    return cfg, D.RuntimeConfig(**base)


@pytest.mark.parametrize("name", list(WORKLOADS))
def test_workspace_sizes(L, name):
    cfg, rt = _cfgs(WORKLOADS[name])
    n = L.dvi_workspace_bytes(ctypes.byref(cfg), ctypes.byref(rt))
    assert n > 0 and n % 256 == 0
    s = WORKLOADS[name].shape
    esz = 2 if WORKLOADS[name].dtype == "bf16" else 4
    kv = 2 * s.n_layers * rt.batch * s.n_kv_heads * rt.max_seq_len * s.head_dim * esz
    assert kv <= n < kv + (1 << 31)


@pytest.mark.parametrize("bad", [dict(k_spec=0), dict(k_spec=17), dict(batch=0), dict(max_seq_len=3),
                                 dict(log_steps=100), dict(max_prefill_chunk=24), dict(head_mode=2),
                                 dict(bonus=2), dict(k_spec=16, bonus=1), dict(persistent=2),
                                 dict(chain_counters=2), dict(megakernel=2)])
def test_invalid_runtime_rejected(L, bad):
    cfg, rt = _cfgs(WORKLOADS["tiny"], **bad)
    assert L.dvi_workspace_bytes(ctypes.byref(cfg), ctypes.byref(rt)) == 0
    ctx = ctypes.c_void_p()
    w = D.WeightsC()
    rc = L.dvi_create(ctypes.byref(cfg), ctypes.byref(rt), ctypes.byref(w), ctypes.c_void_p(256), 1 << 30, None,
                      ctypes.byref(ctx))
    assert rc == -1 and not ctx.value


@pytest.mark.parametrize("name", ["tiny", "7b"])
def test_full_head_mode_workspace(L, name):
    """head_mode 1 adds the Adam moments, the gradient and (bf16) an f32 master of W^(S)."""
    w = WORKLOADS[name]
    cfg, rt0 = _cfgs(w)
    _, rt1 = _cfgs(w, head_mode=1)
    n0 = L.dvi_workspace_bytes(ctypes.byref(cfg), ctypes.byref(rt0))
    n1 = L.dvi_workspace_bytes(ctypes.byref(cfg), ctypes.byref(rt1))
    vd = w.shape.vocab * w.shape.d_model
    per = 16 if w.dtype == "bf16" else 12
    extra = n1 - n0
    assert per * vd <= extra < per * vd + 4 * rt1.log_steps * rt1.batch * rt1.k_spec * w.shape.vocab + 4096


def test_invalid_model_rejected(L):
    cfg, rt = _cfgs(WORKLOADS["tiny"])
    for field, val in (("split_k", 0), ("split_k", 5), ("head_dim", 96), ("d_model", 200), ("n_kv_heads", 3),
                       ("lora_rank", 65), ("dtype", 7)):
        c = D.ModelConfig.from_buffer_copy(cfg)
        setattr(c, field, val)
        assert L.dvi_workspace_bytes(ctypes.byref(c), ctypes.byref(rt)) == 0, field


def test_null_context_calls_fail_cleanly(L):
    assert L.dvi_draft_verify_commit(None, None, None, None) == -1
    assert L.dvi_update_drafter(None, None) == -1
    assert L.dvi_ar_step(None, None) == -1
    assert L.dvi_destroy(None) == -1
    assert L.dvi_last_error(None) == b"null context"


@pytest.mark.parametrize("field", ["final_norm", "lora_b"])
def test_misaligned_vectors_rejected(L, field):
    """final_norm and lora_b are read four floats at a time: dvi_create
    refuses pointers that are not 16-byte aligned, before any device work."""
    cfg, rt = _cfgs(WORKLOADS["tiny"])
    layers = (D.LayerWeightsC * cfg.n_layers)(*[D.LayerWeightsC(*[0x10000] * 9) for _ in range(cfg.n_layers)])
    ptrs = dict(embed=0x20000, final_norm=0x30000, lm_head=0x40000, draft_head=0x40000, lora_a=0x50000,
                lora_b=0x60000)
    ptrs[field] += 4
    w = D.WeightsC(ptrs["embed"], layers, ptrs["final_norm"], ptrs["lm_head"], ptrs["draft_head"], ptrs["lora_a"],
                   ptrs["lora_b"])
    ctx = ctypes.c_void_p()
    rc = L.dvi_create(ctypes.byref(cfg), ctypes.byref(rt), ctypes.byref(w), ctypes.c_void_p(1 << 20), 1 << 30,
                      None, ctypes.byref(ctx))
    assert rc == -1 and not ctx.value


class _FakeTensor:
    """Stands in for a CUDA tensor in the host-side argument checks (no GPU here)."""

    def __init__(self, shape, dtype, device="cuda:0", contiguous=True, cuda=True):
        import torch
        self.shape, self.dtype = tuple(shape), dtype
        self.device = torch.device(device) if cuda else torch.device("cpu")
        self.is_cuda, self._c = cuda, contiguous

    def is_contiguous(self):
        return self._c


def _noalloc_args(**over):
    import torch
    a = dict(w=_FakeTensor((64, 32), torch.bfloat16), x=_FakeTensor((5, 32), torch.float32),
             y=_FakeTensor((5, 64), torch.float32))
    a.update(over)
    return a


def test_noalloc_args_accepted():
    D.check_linear_noalloc_args(**_noalloc_args())


@pytest.mark.parametrize("case", ["x_bf16", "w_f16", "x_short", "y_shape", "rows", "noncontig", "cpu", "devices"])
def test_noalloc_args_rejected_before_any_launch(monkeypatch, case):
    """Every malformed call raises ValueError in the binding, before the
    library is loaded or a pointer reaches the kernel."""
    import torch
    over = {
        "x_bf16": dict(x=_FakeTensor((5, 32), torch.bfloat16)),
        "w_f16": dict(w=_FakeTensor((64, 32), torch.float16)),
        "x_short": dict(x=_FakeTensor((5, 16), torch.float32)),
        "y_shape": dict(y=_FakeTensor((5, 32), torch.float32)),
        "rows": dict(x=_FakeTensor((300, 32), torch.float32), y=_FakeTensor((300, 64), torch.float32)),
        "noncontig": dict(y=_FakeTensor((5, 64), torch.float32, contiguous=False)),
        "cpu": dict(x=_FakeTensor((5, 32), torch.float32, cuda=False)),
        "devices": dict(y=_FakeTensor((5, 64), torch.float32, device="cuda:1")),
    }[case]

    def no_lib():
        raise AssertionError("the library was reached")
    monkeypatch.setattr(D, "lib", no_lib)
    with pytest.raises(ValueError):
        D.linear_noalloc(**_noalloc_args(**over))


@pytest.mark.parametrize("name,takes", [("tiny", False), ("1b", True), ("7b", True), ("7b-b8", False),
                                        ("7b-16k", True)])
def test_megakernel_workspace(L, name, takes):
    """The draft-phase megakernel's scratch (residual, projections, attention
    partials, B u partials, argmax keys, counters, weight and cache
    descriptors) is reserved exactly for the contexts it takes: bf16, at most
    2 sequences, d_ffn a multiple of 64, any context length (tiny: f32;
    7b-b8: 8 sequences; 7b-16k: a 16K context)."""
    w = WORKLOADS[name]
    cfg, rt0 = _cfgs(w, megakernel=0)
    _, rt1 = _cfgs(w, megakernel=1)
    if name == "7b-16k":
        rt0.max_seq_len = rt1.max_seq_len = 16384 + 256
    n0 = L.dvi_workspace_bytes(ctypes.byref(cfg), ctypes.byref(rt0))
    n1 = L.dvi_workspace_bytes(ctypes.byref(cfg), ctypes.byref(rt1))
    assert n0 > 0 and n1 > 0
    if not takes:
        assert n1 == n0
        return
    s = w.shape
    nqkv = (s.n_heads + 2 * s.n_kv_heads) * s.head_dim
    floats = w.batch * (2 * s.d_model + nqkv + 2 * s.d_model + s.d_ffn)   # xr[2], qkv, ao, y, h
    assert n0 + 4 * floats < n1 < n0 + (64 << 20)


def test_megakernel_bf16_small_ffn_not_taken(L):
    """d_ffn must be a multiple of 64 (the weight boxes tile K in 64 columns)."""
    w = WORKLOADS["tiny"].with_(dtype="bf16")
    cfg, rt0 = _cfgs(w, megakernel=0)
    _, rt1 = _cfgs(w, megakernel=1)
    assert w.shape.d_ffn % 64 != 0
    assert L.dvi_workspace_bytes(ctypes.byref(cfg), ctypes.byref(rt1)) == \
        L.dvi_workspace_bytes(ctypes.byref(cfg), ctypes.byref(rt0))


@pytest.mark.parametrize("head_dim,takes", [(64, True), (128, False)])
def test_megakernel_gqa8_only_at_head_dim_64(L, head_dim, takes):
    """A GQA group of 8 goes to the megakernel at head_dim 64 only (at 128 a
    lane's o^T tile of 8 heads would take 64 registers)."""
    shape = tiny_shape(n_layers=4, d_model=16 * head_dim, n_heads=16, n_kv_heads=2, head_dim=head_dim,
                       d_ffn=1408, vocab=4000)
    w = WORKLOADS["tiny"].with_(dtype="bf16", shape=shape)
    cfg, rt0 = _cfgs(w, megakernel=0)
    _, rt1 = _cfgs(w, megakernel=1)
    n0 = L.dvi_workspace_bytes(ctypes.byref(cfg), ctypes.byref(rt0))
    n1 = L.dvi_workspace_bytes(ctypes.byref(cfg), ctypes.byref(rt1))
    assert n0 > 0 and (n1 > n0) == takes and n1 >= n0


@pytest.mark.parametrize("max_seq_len,takes", [(2097087, True), (2097088, False)])
def test_megakernel_cache_rows_below_2_31(L, max_seq_len, takes):
    """The megakernel's key / value boxes address the cache by a 32-bit row
    (layers x sequences x KV heads x max_seq_len, plus 65536 rows of margin
    for a chunk that starts past a full cache): the 7B shape (32 x 1 x 32
    rows per position) is taken up to (2^31 - 1 - 65536) / 1024 = 2097087
    positions."""
    w = WORKLOADS["7b"]
    cfg, rt0 = _cfgs(w, megakernel=0)
    _, rt1 = _cfgs(w, megakernel=1)
    rt0.max_seq_len = rt1.max_seq_len = max_seq_len
    n0 = L.dvi_workspace_bytes(ctypes.byref(cfg), ctypes.byref(rt0))
    n1 = L.dvi_workspace_bytes(ctypes.byref(cfg), ctypes.byref(rt1))
    assert n0 > 0 and (n1 > n0) == takes and n1 >= n0
