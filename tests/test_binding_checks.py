"""The Python binding refuses tensors the C ABI would misread, before any
device call (so these run on the CPU): weights whose shape or dtype differs
from what gf_create copies, host tensors, ids of the wrong type or length,
layouts other than row-major."""
import dataclasses

import pytest

import paper_2605_31464_gb300 as gf
import synth

torch = pytest.importorskip("torch")

SHAPE = dataclasses.replace(synth.SHAPE_TINY, layers=2)


class _FakeCuda(torch.Tensor):
    """A host tensor that reports itself as a CUDA tensor: only the binding's checks look at it."""

    @staticmethod
    def __new__(cls, t):
        return torch.Tensor._make_subclass(cls, t)

    @property
    def is_cuda(self):
        return True


def host_weights(shape, dtype=torch.bfloat16, wrap=_FakeCuda):
    d, hd, L = shape.d_model, shape.head_dim, shape.layers
    z = lambda *s: wrap(torch.zeros(*s, dtype=dtype))
    w = {"embed": z(shape.vocab, d), "lm_head": z(shape.vocab, d), "final_norm": z(d)}
    per = {"attn_norm": (d,), "ffn_norm": (d,), "wq": (shape.n_q * hd, d), "wk": (shape.n_kv * hd, d),
           "wv": (shape.n_kv * hd, d), "wo": (d, shape.n_q * hd), "w_gate": (shape.ffn, d), "w_up": (shape.ffn, d),
           "w_down": (d, shape.ffn)}
    for k, s in per.items():
        w[k] = [z(*s) for _ in range(L)]
    return w


def test_weights_of_the_configured_shapes_pass():
    gf._check_weights(SHAPE, host_weights(SHAPE))


def test_model_refuses_host_weights_before_any_device_call():
    with pytest.raises(ValueError, match="embed: must be a CUDA tensor"):
        gf.Model(SHAPE, host_weights(SHAPE, wrap=lambda t: t), max_batch=2, max_seq=128, max_prefill_tokens=256)


def test_wrong_weight_shape_is_named():
    w = host_weights(SHAPE)
    w["w_down"][1] = _FakeCuda(torch.zeros(SHAPE.ffn, SHAPE.d_model, dtype=torch.bfloat16))  # transposed
    with pytest.raises(ValueError, match=r"w_down\[1\]: shape"):
        gf._check_weights(SHAPE, w)


def test_wrong_weight_dtype_is_refused():
    with pytest.raises(TypeError, match="embed: dtype torch.float32"):
        gf._check_weights(SHAPE, host_weights(SHAPE, torch.float32))


def test_missing_layer_is_refused():
    w = host_weights(SHAPE)
    w["wq"] = w["wq"][:1]
    with pytest.raises(ValueError, match="wq: 1 tensors for 2 layers"):
        gf._check_weights(SHAPE, w)


def test_ids_must_be_int32():
    with pytest.raises(TypeError, match="ids: dtype torch.int64"):
        gf._check_ids(_FakeCuda(torch.zeros(8, dtype=torch.int64)), "ids", 8)


def test_ids_must_cover_the_offsets():
    with pytest.raises(ValueError, match="at least 9 ids"):
        gf._check_ids(_FakeCuda(torch.zeros(8, dtype=torch.int32)), "ids", 9)
    with pytest.raises(ValueError, match="1-D"):
        gf._check_ids(_FakeCuda(torch.zeros(2, 4, dtype=torch.int32)), "ids", 8)
    gf._check_ids(_FakeCuda(torch.zeros(12, dtype=torch.int32)), "ids", 9)  # a longer buffer is fine
    with pytest.raises(ValueError, match="must be a CUDA tensor"):
        gf._check_ids(torch.zeros(12, dtype=torch.int32), "ids", 9)


def test_row_strides_only_where_the_abi_takes_one():
    base = _FakeCuda(torch.zeros(4, 16))
    with pytest.raises(ValueError, match="layout"):
        gf._check_tensor(base.t(), "A", dtype=torch.float32)
    gf._check_tensor(base[:, :8], "logits", dtype=torch.float32, rows_strided=True)
    with pytest.raises(ValueError, match="layout"):
        gf._check_tensor(base[:, ::2], "logits", dtype=torch.float32, rows_strided=True)
