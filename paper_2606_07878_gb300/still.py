"""Thin Python binding of the C ABI in include/still.h (ctypes; argument marshalling only).

Every compute step runs inside libstill.so. Tensors are torch CUDA tensors (device memory and
streams are PyTorch's plumbing); the functions keep the C names. There is no fallback: if the
library is missing or cannot load, every call raises.
"""
from __future__ import annotations

import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libstill.so")

STATUS = {
    0: "STILL_OK", 1: "STILL_ERR_INVALID_ARG", 2: "STILL_ERR_UNSUPPORTED", 3: "STILL_ERR_SHAPE",
    4: "STILL_ERR_ALIGNMENT", 5: "STILL_ERR_NOT_LOADED", 6: "STILL_ERR_OOM", 7: "STILL_ERR_CUDA",
    8: "STILL_ERR_TIMEOUT",
}

# Every entry point include/still.h declares.
EXPORTS = [
    "still_create", "still_destroy", "still_status_string", "still_load_layer_weights",
    "still_compact_layer", "still_compact_stack", "still_compact_layer_ragged",
    "still_compact_stack_ragged", "still_workspace_size", "still_set_workspace_limit",
    "still_set_qhat_eager_limit", "still_profile_enable_classes", "still_reserve_workspace",
    "still_load_layer_weights_blocks",
    "still_get_device_status", "still_budget", "still_kv_bytes", "still_param_count",
    "still_profile_enable", "still_profile_read", "still_kernel_class_name",
    "still_compact_layer_noalloc", "still_recompact_layer_ragged", "still_recompact_stack_ragged",
    "still_selftest_wait_timeout", "still_compact_stack_masked", "still_lookahead_pass_info",
    "still_lookahead_totals", "still_lookahead_compact_layer", "still_lookahead_compact_stack",
    "still_set_beta_head", "still_compact_layer_beta", "still_attend_biased", "still_set_key_fold",
    "still_attend_biased_stack",
]

NOALLOC_SCRATCH_MIB = 64  # STILL_NOALLOC_SCRATCH_MIB in include/still.h

KERNEL_CLASSES = ["strip", "rope_tables", "keyproj", "q_rope", "scores", "softmax", "px",
                  "px_split", "vo", "rmsnorm", "sa_proj", "sa_v", "sa_scores", "sa_softmax",
                  "sa_pv", "sa_out", "ffn1", "ffn2", "heads", "norms", "load", "ca_fused",
                  "beta", "decode", "repair"]


class StillError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        self.name = STATUS.get(code, f"status {code}")
        super().__init__(f"{where}: {self.name}")


class LayerConfig(ctypes.Structure):
    _fields_ = [
        ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
        ("d_latent", ctypes.c_int32), ("n_cross_heads", ctypes.c_int32),
        ("n_self_heads", ctypes.c_int32), ("ffn_dim", ctypes.c_int32),
        ("n_blocks", ctypes.c_int32), ("cross_every_block", ctypes.c_int32),
        ("t_max", ctypes.c_int32), ("final_norm", ctypes.c_int32),
        ("compactor_rope", ctypes.c_int32), ("rope_fix", ctypes.c_int32),
        ("rope_theta", ctypes.c_double), ("rope_theta_compactor", ctypes.c_double),
        ("logit_scale", ctypes.c_double), ("rms_eps", ctypes.c_float), ("l2_eps", ctypes.c_float),
    ]


WEIGHT_NAMES = ["Z", "Wq", "bq", "Wk", "bk", "Wv", "Wo", "Sq", "sbq", "Sk", "sbk", "Sv", "So",
                "W1", "W2", "Wkey", "Wval"]


class LayerWeights(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in WEIGHT_NAMES]


BLOCK_WEIGHT_NAMES = ["Wq", "bq", "Wk", "bk", "Wv", "Wo", "Sq", "sbq", "Sk", "sbk", "Sv", "So",
                      "W1", "W2"]


class BlockWeights(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in BLOCK_WEIGHT_NAMES]


class BetaConfig(ctypes.Structure):
    _fields_ = [("beta_max", ctypes.c_float), ("mass_match", ctypes.c_int32),
                ("log_x", ctypes.c_float)]


class LookaheadPass(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int64) for n in (
        "chunk_start", "chunk_len", "prefill_start", "prefill_len", "prefill_past",
        "compact_row", "retained_after", "logical_after", "pos_offset_after")]


class PosSegment(ctypes.Structure):
    _fields_ = [("start", ctypes.c_double), ("step", ctypes.c_double), ("count", ctypes.c_int64)]


_lib = None


def lib():
    """Loads libstill.so (raises if it is not built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is not built: run __graft_entry__.build()")
        L = ctypes.CDLL(LIB_PATH)
        P, I32, I64, D = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_double
        PI64, PD, PI32 = ctypes.POINTER(I64), ctypes.POINTER(D), ctypes.POINTER(I32)
        PSEG = ctypes.POINTER(PosSegment)
        sig = {
            "still_create": ([ctypes.c_int, ctypes.POINTER(P)], ctypes.c_int),
            "still_destroy": ([P], ctypes.c_int),
            "still_status_string": ([ctypes.c_int], ctypes.c_char_p),
            "still_load_layer_weights_blocks": ([P, I32, ctypes.POINTER(LayerConfig), P,
                                                 ctypes.POINTER(BlockWeights), P, P, P],
                                                ctypes.c_int),
            "still_load_layer_weights": ([P, I32, ctypes.POINTER(LayerConfig),
                                          ctypes.POINTER(LayerWeights), P], ctypes.c_int),
            "still_compact_layer": ([P, I32, P, P, PI64, PSEG, I32, I64, I32, P, P, PD, PD, PI64,
                                     P], ctypes.c_int),
            "still_compact_layer_noalloc": ([P, I32, P, P, PI64, PSEG, I32, I64, I32, P, P, PD,
                                             PD, PI64, P], ctypes.c_int),
            "still_compact_stack": ([P, I32, ctypes.POINTER(P), ctypes.POINTER(P), PI64, PSEG, I32,
                                     I64, I32, ctypes.POINTER(P), ctypes.POINTER(P), PD, PD, PI64,
                                     P], ctypes.c_int),
            "still_compact_layer_ragged": ([P, I32, P, P, PI64, I32, PSEG, PI32, PI32, PI64, P, P,
                                            PI64, P], ctypes.c_int),
            "still_compact_stack_ragged": ([P, I32, ctypes.POINTER(P), ctypes.POINTER(P), PI64, I32,
                                            PSEG, PI32, PI32, PI64, ctypes.POINTER(P),
                                            ctypes.POINTER(P), PI64, P], ctypes.c_int),
            "still_recompact_layer_ragged": ([P, I32, I32, P, P, PI64, PI64, P, P, PI64, I64, P,
                                              P, PI64, PI64, P], ctypes.c_int),
            "still_recompact_stack_ragged": ([P, I32, I32, ctypes.POINTER(P), ctypes.POINTER(P),
                                              PI64, PI64, ctypes.POINTER(P), ctypes.POINTER(P),
                                              PI64, I64, ctypes.POINTER(P), ctypes.POINTER(P),
                                              PI64, PI64, P], ctypes.c_int),
            "still_workspace_size": ([P, I64, I32, ctypes.POINTER(ctypes.c_size_t)], ctypes.c_int),
            "still_set_workspace_limit": ([P, ctypes.c_size_t], ctypes.c_int),
            "still_set_qhat_eager_limit": ([P, ctypes.c_size_t], ctypes.c_int),
            "still_set_key_fold": ([P, I32], ctypes.c_int),
            "still_get_device_status": ([P, P, PI32], ctypes.c_int),
            "still_budget": ([I64, I64], I64),
            "still_kv_bytes": ([I64, I64, I64, I64, I64], I64),
            "still_param_count": ([ctypes.POINTER(LayerConfig), I32], I64),
            "still_selftest_wait_timeout": ([P, I64, P], ctypes.c_int),
            "still_profile_enable": ([P, I32], ctypes.c_int),
            "still_profile_enable_classes": ([P, ctypes.c_uint64], ctypes.c_int),
            "still_reserve_workspace": ([P, I64, I32], ctypes.c_int),
            "still_profile_read": ([P, I32, PI64, PD], ctypes.c_int),
            "still_kernel_class_name": ([I32], ctypes.c_char_p),
            "still_compact_stack_masked": ([P, I32, ctypes.POINTER(ctypes.c_uint8),
                                            ctypes.POINTER(P), ctypes.POINTER(P), PI64, PSEG,
                                            I32, I64, I32, ctypes.POINTER(P), ctypes.POINTER(P),
                                            PD, PD, PI64, P], ctypes.c_int),
            "still_set_beta_head": ([P, I32, P, ctypes.POINTER(BetaConfig), P], ctypes.c_int),
            "still_compact_layer_beta": ([P, I32, P, P, PI64, PSEG, I32, I64, I32, P, P, P, PD,
                                          PD, PI64, P], ctypes.c_int),
            "still_attend_biased": ([P, P, I32, I32, P, P, P, I64, P, P, I64, I32, I32,
                                     ctypes.c_float, P, P], ctypes.c_int),
            "still_attend_biased_stack": ([P, I32, ctypes.POINTER(P), I32, I32,
                                           ctypes.POINTER(P), ctypes.POINTER(P),
                                           ctypes.POINTER(P), I64, ctypes.POINTER(P),
                                           ctypes.POINTER(P), I64, I32, I32, ctypes.c_float,
                                           ctypes.POINTER(P), P], ctypes.c_int),
            "still_lookahead_pass_info": ([I64, I64, I32, ctypes.POINTER(LookaheadPass)],
                                          ctypes.c_int),
            "still_lookahead_totals": ([I64, I64, I32, PI64, PI64], ctypes.c_int),
            "still_lookahead_compact_layer": ([P, I32, I32, P, P, PI64, I64, I32, P, P, P],
                                              ctypes.c_int),
            "still_lookahead_compact_stack": ([P, I32, ctypes.POINTER(ctypes.c_uint8), I32,
                                               ctypes.POINTER(P), ctypes.POINTER(P), PI64, I64,
                                               I32, ctypes.POINTER(P), ctypes.POINTER(P), P],
                                              ctypes.c_int),
        }
        for name, (args, res) in sig.items():
            f = getattr(L, name)
            f.argtypes = args
            f.restype = res
        _lib = L
    return _lib


def _check(code: int, where: str):
    if code != 0:
        raise StillError(code, where)


def _ptr(x):
    if x is None:
        return None
    return ctypes.c_void_p(x.data_ptr())


def _stream(stream):
    if stream is None:
        import torch
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return ctypes.c_void_p(stream)
    return ctypes.c_void_p(stream.cuda_stream)


def _segments(segments):
    if not segments:
        return None, 0
    arr = (PosSegment * len(segments))(*[PosSegment(float(a), float(b), int(c))
                                          for a, b, c in segments])
    return arr, len(segments)


def make_config(H, d, D, n, F, t_max, theta, theta_c=10.0, final_norm=0, logit_scale=0.0,
                rms_eps=1e-6, l2_eps=1e-12, n_blocks=1, cross_every_block=1, compactor_rope=1,
                rope_fix=1) -> LayerConfig:
    return LayerConfig(H, d, D, n, n, F, n_blocks, cross_every_block, t_max, final_norm,
                       compactor_rope, rope_fix, theta, theta_c, logit_scale, rms_eps, l2_eps)


def config_from_workload(wl: dict, t_max: int, **over) -> LayerConfig:
    kw = dict(H=wl["H"], d=wl["d"], D=wl["D"], n=wl["n"], F=wl["F"], t_max=t_max,
              theta=wl["theta"], n_blocks=wl.get("n_blocks", 1),
              cross_every_block=int(wl.get("cross_every_block", 1)),
              compactor_rope=int(wl.get("compactor_rope", 1)))
    kw.update(over)
    return make_config(**kw)


# ------------------------------------------------------------------------------ entry points

def still_status_string(code: int) -> str:
    return lib().still_status_string(code).decode()


def still_create(device: int = 0):
    h = ctypes.c_void_p()
    _check(lib().still_create(device, ctypes.byref(h)), "still_create")
    return h


def still_destroy(ctx):
    _check(lib().still_destroy(ctx), "still_destroy")


def still_set_workspace_limit(ctx, nbytes: int):
    _check(lib().still_set_workspace_limit(ctx, nbytes), "still_set_workspace_limit")


def still_set_qhat_eager_limit(ctx, nbytes: int):
    _check(lib().still_set_qhat_eager_limit(ctx, nbytes), "still_set_qhat_eager_limit")


def still_load_layer_weights(ctx, layer: int, cfg: LayerConfig, weights: dict, stream=None):
    """weights: name -> contiguous bf16 CUDA tensor, layouts as in include/still.h. Block b > 0
    tensors are named "<name>@<b>" (cfg.n_blocks > 1 loads through the per-block entry point)."""
    ptr = lambda name: weights[name].data_ptr() if weights.get(name) is not None else None
    if cfg.n_blocks == 1:
        w = LayerWeights(**{n: ptr(n) for n in WEIGHT_NAMES})
        _check(lib().still_load_layer_weights(ctx, layer, ctypes.byref(cfg), ctypes.byref(w),
                                              _stream(stream)), "still_load_layer_weights")
        return
    blocks = (BlockWeights * cfg.n_blocks)(*[
        BlockWeights(**{n: ptr(n if b == 0 else f"{n}@{b}") for n in BLOCK_WEIGHT_NAMES})
        for b in range(cfg.n_blocks)])
    _check(lib().still_load_layer_weights_blocks(ctx, layer, ctypes.byref(cfg), ptr("Z"), blocks,
                                                 ptr("Wkey"), ptr("Wval"), _stream(stream)),
           "still_load_layer_weights_blocks")


def still_compact_layer(ctx, layer: int, K, V, t: int, Ck, Cv, segments=None, stream=None):
    """K, V [N, H, d] bf16 CUDA (d contiguous); Ck, Cv [t, H, d] bf16 CUDA outputs.
    Returns (out_pos_start, out_pos_step, pos_offset)."""
    strides = (ctypes.c_int64 * 3)(*K.stride())
    assert tuple(V.stride()) == tuple(K.stride()), "K and V must share strides"
    seg, nseg = _segments(segments)
    ps, pst, off = ctypes.c_double(), ctypes.c_double(), ctypes.c_int64()
    _check(lib().still_compact_layer(ctx, layer, _ptr(K), _ptr(V), strides, seg, nseg,
                                     K.shape[0], t, _ptr(Ck), _ptr(Cv), ctypes.byref(ps),
                                     ctypes.byref(pst), ctypes.byref(off), _stream(stream)),
           "still_compact_layer")
    return ps.value, pst.value, off.value


def still_compact_layer_noalloc(ctx, layer: int, K, V, t: int, Ck, Cv, segments=None,
                                stream=None):
    """still_compact_layer without any device allocation (fixed library scratch); same
    arguments and returns."""
    strides = (ctypes.c_int64 * 3)(*K.stride())
    assert tuple(V.stride()) == tuple(K.stride()), "K and V must share strides"
    seg, nseg = _segments(segments)
    ps, pst, off = ctypes.c_double(), ctypes.c_double(), ctypes.c_int64()
    _check(lib().still_compact_layer_noalloc(ctx, layer, _ptr(K), _ptr(V), strides, seg, nseg,
                                             K.shape[0], t, _ptr(Ck), _ptr(Cv),
                                             ctypes.byref(ps), ctypes.byref(pst),
                                             ctypes.byref(off), _stream(stream)),
           "still_compact_layer_noalloc")
    return ps.value, pst.value, off.value


def still_compact_stack(ctx, Ks, Vs, t: int, Cks, Cvs, segments=None, stream=None):
    L = len(Ks)
    P = ctypes.c_void_p
    arr = lambda xs: (P * L)(*[x.data_ptr() for x in xs])
    strides = (ctypes.c_int64 * 3)(*Ks[0].stride())
    seg, nseg = _segments(segments)
    ps, pst, off = ctypes.c_double(), ctypes.c_double(), ctypes.c_int64()
    _check(lib().still_compact_stack(ctx, L, arr(Ks), arr(Vs), strides, seg, nseg,
                                     Ks[0].shape[0], t, arr(Cks), arr(Cvs), ctypes.byref(ps),
                                     ctypes.byref(pst), ctypes.byref(off), _stream(stream)),
           "still_compact_stack")
    return ps.value, pst.value, off.value


def still_compact_stack_masked(ctx, mask, Ks, Vs, t: int, Cks, Cvs, segments=None, stream=None):
    """Compacts the layers l with mask[l] true; the other entries of Ks/Vs/Cks/Cvs may be
    None and are not touched."""
    L = len(mask)
    P = ctypes.c_void_p
    arr = lambda xs: (P * L)(*[(x.data_ptr() if x is not None else None) for x in xs])
    ref = next(k for k, m in zip(Ks, mask) if m)
    strides = (ctypes.c_int64 * 3)(*ref.stride())
    seg, nseg = _segments(segments)
    ps, pst, off = ctypes.c_double(), ctypes.c_double(), ctypes.c_int64()
    m = (ctypes.c_uint8 * L)(*[1 if x else 0 for x in mask])
    _check(lib().still_compact_stack_masked(ctx, L, m, arr(Ks), arr(Vs), strides, seg, nseg,
                                            ref.shape[0], t, arr(Cks), arr(Cvs),
                                            ctypes.byref(ps), ctypes.byref(pst),
                                            ctypes.byref(off), _stream(stream)),
           "still_compact_stack_masked")
    return ps.value, pst.value, off.value


def still_set_beta_head(ctx, layer: int, w_beta, beta_max=0.0, mass_match=0, log_x=0.0,
                        stream=None):
    """w_beta [d_latent] bf16 CUDA tensor; shaping as in include/still.h."""
    bc = BetaConfig(beta_max, mass_match, log_x)
    _check(lib().still_set_beta_head(ctx, layer, _ptr(w_beta), ctypes.byref(bc), _stream(stream)),
           "still_set_beta_head")


def still_compact_layer_beta(ctx, layer: int, K, V, t: int, Ck, Cv, beta, segments=None,
                             stream=None):
    """still_compact_layer plus beta [t, H] fp32; returns (out_pos_start, out_pos_step,
    pos_offset)."""
    strides = (ctypes.c_int64 * 3)(*K.stride())
    assert tuple(V.stride()) == tuple(K.stride()), "K and V must share strides"
    seg, nseg = _segments(segments)
    ps, pst, off = ctypes.c_double(), ctypes.c_double(), ctypes.c_int64()
    _check(lib().still_compact_layer_beta(ctx, layer, _ptr(K), _ptr(V), strides, seg, nseg,
                                          K.shape[0], t, _ptr(Ck), _ptr(Cv), _ptr(beta),
                                          ctypes.byref(ps), ctypes.byref(pst), ctypes.byref(off),
                                          _stream(stream)), "still_compact_layer_beta")
    return ps.value, pst.value, off.value


def still_attend_biased(ctx, q, Ck, Cv, beta, Kfix, Vfix, out, scale=0.0, stream=None):
    """q [nq, Hq, d]; Ck, Cv [t, H, d]; beta [t, H] fp32 or None; Kfix, Vfix [S, H, d];
    out [nq, Hq, d] (bf16 CUDA tensors)."""
    nq, Hq, d = q.shape
    t, H = Ck.shape[0], Ck.shape[1]
    S = Kfix.shape[0]
    _check(lib().still_attend_biased(ctx, _ptr(q), nq, Hq, _ptr(Ck) if t else None,
                                     _ptr(Cv) if t else None, _ptr(beta), t,
                                     _ptr(Kfix) if S else None, _ptr(Vfix) if S else None, S, H,
                                     d, scale, _ptr(out), _stream(stream)), "still_attend_biased")


def still_attend_biased_stack(ctx, q, Ck, Cv, beta, Kfix, Vfix, out, scale=0.0, stream=None):
    """still_attend_biased over a list of layers of one shape, in one launch: q, Ck, Cv, Kfix,
    Vfix, out are lists of per-layer tensors (shapes as in still_attend_biased); beta is None or
    a list whose entries may be None."""
    L = len(q)
    nq, Hq, d = q[0].shape
    t, H = Ck[0].shape[0], Ck[0].shape[1]
    S = Kfix[0].shape[0]
    P = ctypes.c_void_p

    def arr(xs, use=True):
        return (P * L)(*[(x.data_ptr() if use and x is not None else None) for x in xs])

    betas = arr(beta) if beta is not None else None
    _check(lib().still_attend_biased_stack(ctx, L, arr(q), nq, Hq, arr(Ck, t > 0),
                                           arr(Cv, t > 0), betas, t, arr(Kfix, S > 0),
                                           arr(Vfix, S > 0), S, H, d, scale, arr(out),
                                           _stream(stream)), "still_attend_biased_stack")


def still_lookahead_pass_info(k: int, c: int, t: int) -> dict:
    r = LookaheadPass()
    _check(lib().still_lookahead_pass_info(k, c, t, ctypes.byref(r)), "still_lookahead_pass_info")
    return {n: getattr(r, n) for n, _ in LookaheadPass._fields_}


def still_lookahead_totals(T: int, c: int, t: int):
    """(passes, retained cache entries) once T tokens have been compacted."""
    p, r = ctypes.c_int64(), ctypes.c_int64()
    _check(lib().still_lookahead_totals(T, c, t, ctypes.byref(p), ctypes.byref(r)),
           "still_lookahead_totals")
    return p.value, r.value


def still_lookahead_compact_layer(ctx, layer, K, V, passes, c: int, t: int, Ck, Cv,
                                  stream=None):
    """K, V [B*c*t, H, d] packed raw chunks; passes[b] the pass index of sequence b;
    Ck, Cv [B*t, H, d]."""
    B = len(passes)
    _check(lib().still_lookahead_compact_layer(ctx, layer, B, _ptr(K), _ptr(V),
                                               (ctypes.c_int64 * B)(*passes), c, t, _ptr(Ck),
                                               _ptr(Cv), _stream(stream)),
           "still_lookahead_compact_layer")


def still_lookahead_compact_stack(ctx, Ks, Vs, passes, c: int, t: int, Cks, Cvs, mask=None,
                                  stream=None):
    L = len(Ks)
    B = len(passes)
    P = ctypes.c_void_p
    arr = lambda xs: (P * L)(*[(x.data_ptr() if x is not None else None) for x in xs])
    m = None if mask is None else (ctypes.c_uint8 * L)(*[1 if x else 0 for x in mask])
    _check(lib().still_lookahead_compact_stack(ctx, L, m, B, arr(Ks), arr(Vs),
                                               (ctypes.c_int64 * B)(*passes), c, t, arr(Cks),
                                               arr(Cvs), _stream(stream)),
           "still_lookahead_compact_stack")


def _ragged_args(cu_seqlens, ts, segments_per_seq):
    B = len(ts)
    cu = (ctypes.c_int64 * (B + 1))(*cu_seqlens)
    tt = (ctypes.c_int32 * B)(*ts)
    cut = [0]
    for x in ts:
        cut.append(cut[-1] + x)
    cu_t = (ctypes.c_int64 * (B + 1))(*cut)
    if segments_per_seq is None:
        return B, cu, tt, cu_t, None, None
    flat = [s for segs in segments_per_seq for s in segs]
    seg, _ = _segments(flat)
    per = (ctypes.c_int32 * B)(*[len(s) for s in segments_per_seq])
    return B, cu, tt, cu_t, seg, per


def still_compact_layer_ragged(ctx, layer, Kp, Vp, cu_seqlens, ts, Ck, Cv,
                               segments_per_seq=None, stream=None):
    """Kp, Vp [sum N_b, H, d]; Ck, Cv [sum t_b, H, d]. Returns the per-sequence offsets."""
    B, cu, tt, cu_t, seg, per = _ragged_args(cu_seqlens, ts, segments_per_seq)
    off = (ctypes.c_int64 * B)()
    _check(lib().still_compact_layer_ragged(ctx, layer, _ptr(Kp), _ptr(Vp), cu, B, seg, per, tt,
                                            cu_t, _ptr(Ck), _ptr(Cv), off, _stream(stream)),
           "still_compact_layer_ragged")
    return list(off)


def still_compact_stack_ragged(ctx, Kps, Vps, cu_seqlens, ts, Cks, Cvs, segments_per_seq=None,
                               stream=None):
    L = len(Kps)
    P = ctypes.c_void_p
    arr = lambda xs: (P * L)(*[x.data_ptr() for x in xs])
    B, cu, tt, cu_t, seg, per = _ragged_args(cu_seqlens, ts, segments_per_seq)
    off = (ctypes.c_int64 * B)()
    _check(lib().still_compact_stack_ragged(ctx, L, arr(Kps), arr(Vps), cu, B, seg, per, tt, cu_t,
                                            arr(Cks), arr(Cvs), off, _stream(stream)),
           "still_compact_stack_ragged")
    return list(off)


def still_recompact_layer_ragged(ctx, layer, Kprev, Vprev, cu_prev, prev_len, Knew, Vnew,
                                 cu_new, ratio, Ck, Cv, stream=None):
    """[previous compact | new tokens] -> new compact caches. Returns (cu_out, len_out)."""
    B = len(prev_len)
    I64 = ctypes.c_int64
    cu_out = (I64 * (B + 1))()
    len_out = (I64 * B)()
    _check(lib().still_recompact_layer_ragged(
        ctx, layer, B, _ptr(Kprev), _ptr(Vprev), (I64 * (B + 1))(*cu_prev), (I64 * B)(*prev_len),
        _ptr(Knew), _ptr(Vnew), (I64 * (B + 1))(*cu_new), ratio, _ptr(Ck), _ptr(Cv), cu_out,
        len_out, _stream(stream)), "still_recompact_layer_ragged")
    return list(cu_out), list(len_out)


def still_recompact_stack_ragged(ctx, Kprevs, Vprevs, cu_prev, prev_len, Knews, Vnews, cu_new,
                                 ratio, Cks, Cvs, stream=None):
    L = len(Kprevs)
    B = len(prev_len)
    P, I64 = ctypes.c_void_p, ctypes.c_int64
    arr = lambda xs: (P * L)(*[x.data_ptr() for x in xs])
    cu_out = (I64 * (B + 1))()
    len_out = (I64 * B)()
    _check(lib().still_recompact_stack_ragged(
        ctx, L, B, arr(Kprevs), arr(Vprevs), (I64 * (B + 1))(*cu_prev), (I64 * B)(*prev_len),
        arr(Knews), arr(Vnews), (I64 * (B + 1))(*cu_new), ratio, arr(Cks), arr(Cvs), cu_out,
        len_out, _stream(stream)), "still_recompact_stack_ragged")
    return list(cu_out), list(len_out)


def still_set_key_fold(ctx, enable: bool):
    _check(lib().still_set_key_fold(ctx, 1 if enable else 0), "still_set_key_fold")


def still_reserve_workspace(ctx, max_tokens: int, max_t: int):
    _check(lib().still_reserve_workspace(ctx, max_tokens, max_t), "still_reserve_workspace")


def still_workspace_size(ctx, max_tokens: int, max_t: int) -> int:
    b = ctypes.c_size_t()
    _check(lib().still_workspace_size(ctx, max_tokens, max_t, ctypes.byref(b)),
           "still_workspace_size")
    return b.value


def still_get_device_status(ctx, stream=None):
    """Synchronizes the stream; returns (status_code, [code, site, block, count])."""
    det = (ctypes.c_int32 * 4)()
    code = lib().still_get_device_status(ctx, _stream(stream), det)
    return code, list(det)


def still_budget(n_tokens: int, ratio: int) -> int:
    return lib().still_budget(n_tokens, ratio)


def still_kv_bytes(L, H, d, b, S) -> int:
    return lib().still_kv_bytes(L, H, d, b, S)


def still_param_count(cfg: LayerConfig, t: int) -> int:
    return lib().still_param_count(ctypes.byref(cfg), t)


def still_profile_enable(ctx, enable: bool = True):
    _check(lib().still_profile_enable(ctx, 1 if enable else 0), "still_profile_enable")


def still_profile_enable_classes(ctx, names):
    """Event timing only for the named kernel classes (an empty list stops timing)."""
    mask = 0
    for n in names:
        mask |= 1 << KERNEL_CLASSES.index(n)
    _check(lib().still_profile_enable_classes(ctx, mask), "still_profile_enable_classes")


def still_profile_read(ctx):
    """{class name: (launches, total ms)} since the last still_profile_enable."""
    out = {}
    for i, name in enumerate(KERNEL_CLASSES):
        n, ms = ctypes.c_int64(), ctypes.c_double()
        _check(lib().still_profile_read(ctx, i, ctypes.byref(n), ctypes.byref(ms)),
               "still_profile_read")
        out[name] = (n.value, ms.value)
    return out


def still_kernel_class_name(cls: int) -> str:
    return lib().still_kernel_class_name(cls).decode()


def still_selftest_wait_timeout(ctx, limit_us: int = 1000, stream=None):
    _check(lib().still_selftest_wait_timeout(ctx, limit_us, _stream(stream)),
           "still_selftest_wait_timeout")
