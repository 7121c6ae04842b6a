"""The C-ABI library builds, loads and exports every declared symbol; host-only
entry points work without a GPU (no compute calls here)."""
import ctypes
import os
import re

import pytest

import oracle_pins as P

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2609_35701_gb300 import build

    path = build.build()
    return ctypes.CDLL(path)


def declared_symbols():
    with open(os.path.join(ROOT, "include", "meq.h")) as f:
        text = f.read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(meq_[a-z_0-9]+)\s*\(", text)))


def test_every_declared_symbol_is_exported(lib):
    names = declared_symbols()
    assert len(names) >= 14
    for n in names:
        assert hasattr(lib, n), n


def test_binding_covers_the_header():
    from paper_2609_35701_gb300 import meq

    assert sorted(meq.EXPORTED) == declared_symbols()


def test_default_options_are_the_papers():
    from paper_2609_35701_gb300 import meq

    o = meq.default_options()
    g = P.golden()
    assert abs(o.ns_a - g["ns"]["a"]) < 1e-6 and abs(o.ns_b - g["ns"]["b"]) < 1e-6 and abs(o.ns_c - g["ns"]["c"]) < 1e-6
    assert o.ns_steps == g["ns"]["steps"] and abs(o.rho - g["rho"]) < 1e-7
    assert o.nesterov == 0 and o.use_graph == 1
    assert o.ns_cta_pair == 1 and o.ns_x0_fused == 1 and o.update_rule == meq.RULE_MEQMUON


def test_state_holds_momentum_only():
    """Section 4 'Memory overhead': MeqMuon keeps one fp32 momentum value per
    element of the hidden weights (no second moment, no per-row state)."""
    from paper_2609_35701_gb300 import meq, workloads as W

    g = P.golden()["architecture"]
    for wl, arch in (("llama130m", "Llama-130M"), ("llama350m", "Llama-350M")):
        shapes = [(r, c) for _, r, c in W.get_workload(wl).shapes]
        persistent, workspace = meq.state_bytes(shapes)
        Nh, _ = P.llama_hidden_counts(g[arch])
        assert persistent == 4 * Nh
        assert workspace > 0


def test_full_model_state_reproduces_table5():
    """Algorithm 1 over every trainable parameter keeps one fp32 momentum value
    per parameter: the library's persistent bytes for the full Table 11 models
    equal the MeqMuon column of Table 5 (Section 4, 'Memory overhead')."""
    from paper_2609_35701_gb300 import meq, workloads as W

    g = P.golden()
    for name, a in g["architecture"].items():
        params = W.full_model_params(a["layers"], a["hidden"], a["ffn"], a["vocab"], a["q_heads"], a["kv_heads"],
                                     a["head_dim"], tied=a["tied"], qkv_bias=name.startswith("Qwen2"))
        assert abs(sum(r * c for _, r, c, _ in params) / 1e6 - a["params_m"]) < 5e-4, name
        persistent, _ = meq.state_bytes([(r, c) for _, r, c, _ in params], kinds=[k for _, _, _, k in params])
        assert round(persistent / 2 ** 20, 2) == g["state_mib"]["MeqMuon"][name], name


def test_kind_validation():
    from paper_2609_35701_gb300 import meq

    with pytest.raises(meq.MeqError) as e:
        meq.state_bytes([(2, 8)], kinds=[meq.VECTOR])   # vectors are (1, d)
    assert e.value.status == 1
    with pytest.raises(meq.MeqError):
        meq.state_bytes([(2, 8)], kinds=[7])


def test_host_validation_errors():
    from paper_2609_35701_gb300 import meq

    for bad in ([], [(0, 4)], [(3, -1)], [(1 << 21, 2)]):
        with pytest.raises(meq.MeqError) as e:
            meq.state_bytes(bad)
        assert e.value.status == 1
    with pytest.raises(meq.MeqError):
        meq.state_bytes([(4, 4)], ns_steps=0)
    # the size limits, at and just past their edges (dims 2^20, elements 2^34)
    meq.state_bytes([(1 << 20, 1), (1, 1 << 20), (1 << 20, 1 << 14)])
    for bad in ([(1 << 20, (1 << 14) + 1)], [((1 << 20) + 1, 1)], [(1, (1 << 20) + 1)]):
        with pytest.raises(meq.MeqError) as e:
            meq.state_bytes(bad)
        assert e.value.status == 1
    p0, w0 = meq.state_bytes([(300, 200), (1, 64)], kinds=[meq.HIDDEN, meq.VECTOR])
    p1, w1 = meq.state_bytes([(300, 200), (1, 64)], kinds=[meq.HIDDEN, meq.VECTOR], debug_canaries=1)
    assert p1 == p0 and w1 > w0  # guard bands are workspace only
    for field in ("ns_cta_pair", "ns_x0_fused", "update_rule", "debug_canaries", "debug_skip_load"):
        with pytest.raises(meq.MeqError):
            meq.state_bytes([(4, 4)], **{field: 2})
    # Eq. (6) is the hidden-weight baseline only
    meq.state_bytes([(4, 4)], update_rule=meq.RULE_MUON)
    with pytest.raises(meq.MeqError) as e:
        meq.state_bytes([(4, 4), (1, 4)], kinds=[meq.HIDDEN, meq.VECTOR], update_rule=meq.RULE_MUON)
    assert e.value.status == 1


def test_binding_rejects_tensors_the_library_cannot_check(lib):
    """The library sees raw pointers only; the binding refuses host tensors,
    other dtypes, strided views and wrong element counts before any call."""
    import torch

    from paper_2609_35701_gb300 import meq

    for t, dt, n in [(torch.zeros(4, 4), "float32", 16),                     # host memory
                     (torch.zeros(4, 4, dtype=torch.float64), "float32", 16)]:
        with pytest.raises(ValueError):
            meq._require_cuda(t, dt, n, "x")
    H = torch.zeros(8, 8)
    with pytest.raises(ValueError):
        meq.ns_cv_trajectory(H)
    with pytest.raises(ValueError):
        meq.row_col_stats_noalloc(H, torch.zeros(8), torch.zeros(8), torch.zeros(2, dtype=torch.float64),
                                  torch.zeros(1, dtype=torch.int32))


def test_noalloc_size_checks_come_before_any_cuda_call():
    """meq_row_col_stats_noalloc refuses bad arguments and shapes beyond its
    fixed scratch on the host, with a message, before it looks for a device:
    here, with no GPU at all, every refusal is MEQ_ERR_INVALID_ARG (a call
    that got as far as the device would return MEQ_ERR_CUDA instead)."""
    from paper_2609_35701_gb300 import meq

    fn = meq.lib.meq_row_col_stats_noalloc
    fake = 4096  # never dereferenced: the checks are host-only
    cases = [
        (fake, 8192, 8192, 1e-7, 1e-6, b"scratch"),          # 8192 * 8 + 256 * 8192 floats > 2^21
        (fake, 1 << 20, 1 << 12, 1e-7, 1e-6, b"scratch"),
        (fake, (1 << 20) + 1, 4, 1e-7, 1e-6, b"rows and cols"),
        (fake, 0, 4, 1e-7, 1e-6, b"rows and cols"),
        (None, 4, 4, 1e-7, 1e-6, b"NULL"),
        (fake, 4, 4, -1.0, 1e-6, b"eps"),
    ]
    for U, m, n, eps, tie, text in cases:
        assert fn(U, m, n, eps, tie, fake, fake, fake, fake, None) == 1, (m, n)
        assert text in meq.lib.meq_last_error(None), (m, n, meq.lib.meq_last_error(None))
    # the largest Llama-7B hidden shapes fit: 11008 * 4 + 344 * 4096 and 4096 * 11 + 128 * 11008 floats
    assert 11008 * 4 + 344 * 4096 <= 1 << 21 and 4096 * 11 + 128 * 11008 <= 1 << 21
