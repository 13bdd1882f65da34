"""Thin ctypes binding of the OUTLETS C ABI (include/outlets.h).

Argument marshalling only: every step of the forward runs in the CUDA library.
PyTorch supplies device memory and streams.  If the library is missing the
binding raises; there is no other code path.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "liboutlets_gb300.so")
MAX_HEAD_HIDDEN = 7

OK, EINVAL, ENOMEM, ECUDA, EUNSUPPORTED, ECAPACITY, ETIMEOUT, EDEVICE = range(8)
STATUS_NAMES = ["OK", "EINVAL", "ENOMEM", "ECUDA", "EUNSUPPORTED", "ECAPACITY", "ETIMEOUT", "EDEVICE"]
F32, BF16 = 0, 1
ALL_TOKENS = 1
KEEP_ROWS = 2
T_FCTX, T_XIN, T_Q, T_ATTN, T_A, T_Y, T_HDRAFT = range(7)
N_STAGES = 12
MAX_TOPK = 8

c_i32, c_f32, c_vp = ctypes.c_int32, ctypes.c_float, ctypes.c_void_p


class Config(ctypes.Structure):
    _fields_ = [("d_model", c_i32), ("n_heads", c_i32), ("n_kv_heads", c_i32), ("head_dim", c_i32),
                ("ffn_dim", c_i32), ("n_head_hidden", c_i32), ("head_hidden", c_i32 * MAX_HEAD_HIDDEN),
                ("rope_theta", c_f32), ("rms_eps", c_f32), ("dtype", c_i32), ("max_tokens", c_i32),
                ("max_batch", c_i32), ("max_position", c_i32), ("device", c_i32), ("vocab", c_i32),
                ("embed_vocab", c_i32)]


_WNAMES = ["w_proj", "w_q", "w_k", "w_v", "w_o", "g_in", "g_post", "g_final", "w_gate", "w_up", "w_down"]


class Weights(ctypes.Structure):
    _fields_ = [(n, c_vp) for n in _WNAMES] + [("head_w", c_vp * (MAX_HEAD_HIDDEN + 1)),
                                               ("head_b", c_vp * (MAX_HEAD_HIDDEN + 1)),
                                               ("w_attn_gate", c_vp), ("w_lm", c_vp), ("w_embed", c_vp),
                                               ("g_emb", c_vp)]


class DraftOut(ctypes.Structure):
    _fields_ = [("k", c_i32), ("topk_ids", c_vp), ("topk_logprob", c_vp), ("logsumexp", c_vp), ("logits", c_vp)]


class SchedConfig(ctypes.Structure):
    _fields_ = [("n_decode", c_i32), ("max_running", c_i32), ("route", c_i32), ("order", c_i32),
                ("pf_base_s", ctypes.c_double), ("pf_per_token_s", ctypes.c_double),
                ("step_base_s", ctypes.c_double), ("step_per_seq_s", ctypes.c_double),
                ("step_per_kv_token_s", ctypes.c_double)]


ROUTE_RR, ROUTE_LB = 0, 1
ORDER_FCFS, ORDER_SJF = 0, 1


class TensorInfo(ctypes.Structure):
    _fields_ = [("dtype", c_i32), ("rows", c_i32), ("cols", c_i32)]


class OutletsError(RuntimeError):
    def __init__(self, status, msg):
        self.status = status
        super().__init__(f"{STATUS_NAMES[status] if 0 <= status < 8 else status}: {msg}")


_lib = None


def load():
    """Load the CUDA library (built by ``paper_2609_01068_gb300.build``)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: run `python -m paper_2609_01068_gb300.build` first")
    lib = ctypes.CDLL(LIB_PATH)
    P = ctypes.POINTER
    sig = {
        "outlets_create": (c_i32, [P(Config), P(Weights), P(c_vp)]),
        "outlets_destroy": (None, [c_vp]),
        "outlets_last_error": (ctypes.c_char_p, [c_vp]),
        "outlets_device_bytes": (ctypes.c_size_t, [c_vp]),
        "outlets_kv_create": (c_i32, [c_vp, c_i32, c_i32, P(c_vp)]),
        "outlets_kv_destroy": (None, [c_vp]),
        "outlets_kv_reset_slot": (c_i32, [c_vp, c_i32]),
        "outlets_kv_slot_length": (c_i32, [c_vp, c_i32]),
        "outlets_kv_free_pages": (c_i32, [c_vp]),
        "outlets_predict_prefill": (c_i32, [c_vp, P(c_vp), c_vp, c_i32, c_i32, c_vp, c_vp, ctypes.c_uint32,
                                            c_vp, c_vp, c_vp]),
        "outlets_predict_step": (c_i32, [c_vp, P(c_vp), c_i32, c_vp, c_vp, c_vp, c_vp, c_vp]),
        "outlets_predict_prefill_dual": (c_i32, [c_vp, P(c_vp), c_vp, c_i32, c_i32, c_vp, c_vp, ctypes.c_uint32,
                                                 c_vp, c_vp, P(DraftOut), c_vp]),
        "outlets_predict_step_dual": (c_i32, [c_vp, P(c_vp), c_i32, c_vp, c_vp, c_vp, c_vp, P(DraftOut), c_vp]),
        "outlets_draft_head": (c_i32, [c_vp, c_vp, c_i32, P(DraftOut), c_vp]),
        "outlets_predict_prefill_ex": (c_i32, [c_vp, P(c_vp), c_vp, c_vp, c_i32, c_i32, c_vp, c_vp, ctypes.c_uint32,
                                               c_vp, c_vp, c_vp, c_vp]),
        "outlets_predict_step_ex": (c_i32, [c_vp, P(c_vp), c_vp, c_i32, c_vp, c_vp, c_vp, c_vp, c_vp, c_vp]),
        "outlets_predict_draft_step": (c_i32, [c_vp, c_vp, c_i32, c_vp, c_vp, c_vp, c_vp, c_vp, c_vp]),
        "outlets_kv_truncate": (c_i32, [c_vp, c_i32, c_i32]),
        "outlets_check": (c_i32, [c_vp, c_vp]),
        "outlets_get_intermediate": (c_i32, [c_vp, c_i32, c_vp, ctypes.c_size_t, P(TensorInfo), c_vp]),
        "outlets_profile_enable": (c_i32, [c_vp, c_i32]),
        "outlets_profile_read": (c_i32, [c_vp, P(ctypes.c_double), P(c_i32)]),
        "outlets_stage_name": (ctypes.c_char_p, [c_i32]),
        "outlets_launch_count": (ctypes.c_uint64, [c_vp]),
        "outlets_length_head_noalloc": (c_i32, [c_vp, c_vp, c_i32, c_vp, c_vp, c_vp]),
        "outlets_selftest_bounded_wait": (c_i32, [c_vp, ctypes.c_uint64, c_vp]),
        "outlets_sched_simulate": (c_i32, [P(SchedConfig), c_i32, c_vp, c_vp, c_vp, c_vp, c_vp, c_vp]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def _ptr(x):
    """Address of a torch tensor or a numpy array (None -> NULL)."""
    if x is None:
        return None
    if isinstance(x, np.ndarray):
        if not x.flags["C_CONTIGUOUS"]:
            raise ValueError("arrays must be C-contiguous")
        return x.ctypes.data
    if not x.is_contiguous():
        raise ValueError("tensors must be contiguous")
    return x.data_ptr()


def _tokens(tokens):
    """Token ids as a contiguous int32 array/tensor (device tensors stay on the device)."""
    if isinstance(tokens, np.ndarray) or not hasattr(tokens, "data_ptr"):
        return np.ascontiguousarray(tokens, dtype=np.int32)
    import torch
    return tokens.to(torch.int32).contiguous()


def _stream_handle(stream):
    import torch
    if stream is None:
        return torch.cuda.current_stream().cuda_stream if torch.cuda.is_available() else 0
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


class Predictor:
    """One OUTLETS draft backbone + length head resident on a GPU."""

    def __init__(self, shape, weights: dict, max_tokens: int, max_batch: int, max_position: int = 16384,
                 device: int = 0):
        self.lib = load()
        self.shape = shape
        cfg = Config()
        cfg.d_model, cfg.n_heads, cfg.n_kv_heads = shape.d, shape.n_heads, shape.n_kv_heads
        cfg.head_dim, cfg.ffn_dim = shape.head_dim, shape.ffn
        cfg.n_head_hidden = len(shape.head_widths)
        for i, wdt in enumerate(shape.head_widths):
            cfg.head_hidden[i] = wdt
        cfg.rope_theta, cfg.rms_eps = shape.rope_theta, shape.rms_eps
        cfg.dtype = BF16 if shape.dtype == "bf16" else F32
        cfg.max_tokens, cfg.max_batch, cfg.max_position, cfg.device = max_tokens, max_batch, max_position, device
        self.cfg = cfg
        self.device = device
        keep = {}
        w = Weights()
        for n in _WNAMES:
            a = np.ascontiguousarray(weights[n], dtype=np.float32)
            keep[n] = a
            setattr(w, n, a.ctypes.data)
        for i in range(len(shape.head_widths) + 1):
            wa = np.ascontiguousarray(weights[f"head_w{i}"], dtype=np.float32)
            ba = np.ascontiguousarray(weights[f"head_b{i}"], dtype=np.float32)
            keep[f"hw{i}"], keep[f"hb{i}"] = wa, ba
            w.head_w[i] = wa.ctypes.data
            w.head_b[i] = ba.ctypes.data
        if weights.get("w_attn_gate") is not None:  # gated attention
            ga = np.ascontiguousarray(weights["w_attn_gate"], dtype=np.float32)
            keep["w_attn_gate"] = ga
            w.w_attn_gate = ga.ctypes.data
        if weights.get("w_lm") is not None:  # draft LM head of the dual head (Eq. 2)
            la = np.ascontiguousarray(weights["w_lm"], dtype=np.float32)
            keep["w_lm"] = la
            w.w_lm = la.ctypes.data
            cfg.vocab = la.shape[0]
        self.vocab = cfg.vocab
        if weights.get("w_embed") is not None:  # input-embedding branch
            ea = np.ascontiguousarray(weights["w_embed"], dtype=np.float32)
            ga = np.ascontiguousarray(weights["g_emb"], dtype=np.float32)
            keep["w_embed"], keep["g_emb"] = ea, ga
            w.w_embed, w.g_emb = ea.ctypes.data, ga.ctypes.data
            cfg.embed_vocab = ea.shape[0]
        self.embed_vocab = cfg.embed_vocab
        h = c_vp()
        st = self.lib.outlets_create(ctypes.byref(cfg), ctypes.byref(w), ctypes.byref(h))
        if st != OK:
            raise OutletsError(st, "outlets_create failed")
        self.h = h

    # -- helpers
    def _raise(self, st):
        msg = self.lib.outlets_last_error(self.h)
        raise OutletsError(st, msg.decode() if msg else "")

    def close(self):
        if getattr(self, "h", None):
            self.lib.outlets_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    @property
    def device_bytes(self):
        return self.lib.outlets_device_bytes(self.h)

    def _outputs(self, n, like, z_out, len_out):
        import torch
        if z_out is None:
            dev = like.device if hasattr(like, "device") else torch.device("cpu")
            z_out = torch.empty(n, dtype=torch.float32, device=dev)
            len_out = torch.empty(n, dtype=torch.float32, device=dev)
        return z_out, len_out

    # -- prediction
    def prefill(self, taps, cu_seqlens, kv=None, slots=None, all_tokens=False, z_out=None, len_out=None,
                stream=None, tokens=None, keep_rows=False):
        """Static prediction (z_hat, length_hat) for a packed varlen batch.
        tokens: [T] int32 ids (numpy or torch), for the input-embedding branch.
        keep_rows: run the whole layer on every row (keeps every row's
        intermediates); otherwise only the predicted rows go past the K/V."""
        cu = np.ascontiguousarray(cu_seqlens, dtype=np.int32)
        B, T = len(cu) - 1, int(cu[-1]) if len(cu) else 0
        n_out = T if all_tokens else B
        z_out, len_out = self._outputs(n_out, taps[0], z_out, len_out)
        tp = (c_vp * 3)(*[_ptr(t) for t in taps])
        sl = None if slots is None else np.ascontiguousarray(slots, dtype=np.int32)
        args = (cu.ctypes.data, B, T, kv.h if kv else None, None if sl is None else sl.ctypes.data,
                (ALL_TOKENS if all_tokens else 0) | (KEEP_ROWS if keep_rows else 0), _ptr(z_out), _ptr(len_out))
        if tokens is None:
            st = self.lib.outlets_predict_prefill(self.h, tp, *args, _stream_handle(stream))
        else:
            tok = _tokens(tokens)
            st = self.lib.outlets_predict_prefill_ex(self.h, tp, _ptr(tok), *args, None, _stream_handle(stream))
        if st != OK:
            self._raise(st)
        return z_out, len_out

    def step(self, taps, kv, slots, z_out=None, len_out=None, stream=None, tokens=None):
        """Dynamic prediction for one new token per request (tokens: their ids, [B])."""
        sl = np.ascontiguousarray(slots, dtype=np.int32)
        B = len(sl)
        z_out, len_out = self._outputs(B, taps[0], z_out, len_out)
        tp = (c_vp * 3)(*[_ptr(t) for t in taps])
        if tokens is None:
            st = self.lib.outlets_predict_step(self.h, tp, B, kv.h, sl.ctypes.data, _ptr(z_out), _ptr(len_out),
                                               _stream_handle(stream))
        else:
            tok = _tokens(tokens)
            st = self.lib.outlets_predict_step_ex(self.h, tp, _ptr(tok), B, kv.h, sl.ctypes.data, _ptr(z_out),
                                                  _ptr(len_out), None, _stream_handle(stream))
        if st != OK:
            self._raise(st)
        return z_out, len_out

    # -- dual head (Sec. 4.2, Eq. 2)
    def _draft_out(self, n, k, like, logits, out=None):
        """DraftOut for n rows: torch outputs on like's device unless `out` supplies them."""
        import torch
        if out is None:
            dev = like.device if hasattr(like, "device") else torch.device("cpu")
            out = {"ids": torch.empty((n, k), dtype=torch.int32, device=dev),
                   "logprob": torch.empty((n, k), dtype=torch.float32, device=dev),
                   "lse": torch.empty(n, dtype=torch.float32, device=dev)}
            if logits:
                out["logits"] = torch.empty((n, self.vocab), dtype=torch.float32, device=dev)
        d = DraftOut()
        d.k = k
        d.topk_ids, d.topk_logprob = _ptr(out["ids"]), _ptr(out["logprob"])
        d.logsumexp, d.logits = _ptr(out.get("lse")), _ptr(out.get("logits"))
        return d, out

    def prefill_dual(self, taps, cu_seqlens, k, kv=None, slots=None, all_tokens=False, logits=False, out=None,
                     z_out=None, len_out=None, stream=None, tokens=None, keep_rows=False):
        """Static prediction plus the draft head on the same rows:
        (z_hat, length_hat, {"ids", "logprob", "lse"[, "logits"]})."""
        cu = np.ascontiguousarray(cu_seqlens, dtype=np.int32)
        B, T = len(cu) - 1, int(cu[-1]) if len(cu) else 0
        n_out = T if all_tokens else B
        z_out, len_out = self._outputs(n_out, taps[0], z_out, len_out)
        d, draft = self._draft_out(n_out, k, taps[0], logits, out)
        tp = (c_vp * 3)(*[_ptr(t) for t in taps])
        sl = None if slots is None else np.ascontiguousarray(slots, dtype=np.int32)
        args = (cu.ctypes.data, B, T, kv.h if kv else None, None if sl is None else sl.ctypes.data,
                (ALL_TOKENS if all_tokens else 0) | (KEEP_ROWS if keep_rows else 0), _ptr(z_out), _ptr(len_out),
                ctypes.byref(d))
        if tokens is None:
            st = self.lib.outlets_predict_prefill_dual(self.h, tp, *args, _stream_handle(stream))
        else:
            tok = _tokens(tokens)
            st = self.lib.outlets_predict_prefill_ex(self.h, tp, _ptr(tok), *args, _stream_handle(stream))
        if st != OK:
            self._raise(st)
        return z_out, len_out, draft

    def step_dual(self, taps, kv, slots, k, logits=False, out=None, z_out=None, len_out=None, stream=None,
                  tokens=None):
        """Dynamic prediction plus the draft head: (z_hat, length_hat, draft outputs)."""
        sl = np.ascontiguousarray(slots, dtype=np.int32)
        B = len(sl)
        z_out, len_out = self._outputs(B, taps[0], z_out, len_out)
        d, draft = self._draft_out(B, k, taps[0], logits, out)
        tp = (c_vp * 3)(*[_ptr(t) for t in taps])
        if tokens is None:
            st = self.lib.outlets_predict_step_dual(self.h, tp, B, kv.h, sl.ctypes.data, _ptr(z_out), _ptr(len_out),
                                                    ctypes.byref(d), _stream_handle(stream))
        else:
            tok = _tokens(tokens)
            st = self.lib.outlets_predict_step_ex(self.h, tp, _ptr(tok), B, kv.h, sl.ctypes.data, _ptr(z_out),
                                                  _ptr(len_out), ctypes.byref(d), _stream_handle(stream))
        if st != OK:
            self._raise(st)
        return z_out, len_out, draft

    def draft_head(self, h_draft, k, logits=False, out=None, stream=None):
        """The draft head alone on device states h_draft [rows, d]."""
        rows = int(h_draft.shape[0])
        d, draft = self._draft_out(rows, k, h_draft, logits, out)
        st = self.lib.outlets_draft_head(self.h, _ptr(h_draft), rows, ctypes.byref(d), _stream_handle(stream))
        if st != OK:
            self._raise(st)
        return draft

    def draft_step(self, kv, slots, tokens=None, k=None, logits=False, out=None, z_out=None, len_out=None,
                   stream=None):
        """One draft rollout position per request, fed by the previous step's own output
        state: (z_hat, length_hat) or, with k, (z_hat, length_hat, draft outputs)."""
        sl = np.ascontiguousarray(slots, dtype=np.int32)
        B = len(sl)
        like = tokens if tokens is not None and hasattr(tokens, "device") else z_out
        if like is None:
            import torch
            like = torch.empty(0, device=f"cuda:{self.device}")
        z_out, len_out = self._outputs(B, like, z_out, len_out)
        d, draft = (self._draft_out(B, k, like, logits, out) if k else (None, None))
        tok = None if tokens is None else _tokens(tokens)
        st = self.lib.outlets_predict_draft_step(self.h, _ptr(tok), B, kv.h, sl.ctypes.data, _ptr(z_out),
                                                 _ptr(len_out), ctypes.byref(d) if d is not None else None,
                                                 _stream_handle(stream))
        if st != OK:
            self._raise(st)
        return (z_out, len_out, draft) if k else (z_out, len_out)

    def selftest_bounded_wait(self, timeout_ns=1_000_000, stream=None):
        """Enqueue a kernel whose bounded wait runs out (see outlets_check)."""
        st = self.lib.outlets_selftest_bounded_wait(self.h, timeout_ns, _stream_handle(stream))
        if st != OK:
            self._raise(st)

    def check(self, stream=None):
        st = self.lib.outlets_check(self.h, _stream_handle(stream))
        if st != OK:
            self._raise(st)

    def profile(self, enable, stages=None):
        """Time the named stages (all if None) of later calls; enable=False turns timing off."""
        mask = 0
        if enable:
            if stages is None:
                mask = -1
            else:
                names = [self.lib.outlets_stage_name(i).decode() for i in range(N_STAGES)]
                for n in stages:
                    mask |= 1 << names.index(n)
        st = self.lib.outlets_profile_enable(self.h, mask)
        if st != OK:
            self._raise(st)

    def profile_read(self):
        """{stage name: (total ms, runs)} of the calls since profiling was enabled / last read."""
        ms = (ctypes.c_double * N_STAGES)()
        cnt = (c_i32 * N_STAGES)()
        st = self.lib.outlets_profile_read(self.h, ms, cnt)
        if st != OK:
            self._raise(st)
        return {self.lib.outlets_stage_name(i).decode(): (ms[i], cnt[i]) for i in range(N_STAGES)}

    @property
    def launch_count(self):
        return int(self.lib.outlets_launch_count(self.h))

    def intermediate(self, which, stream=None):
        """Copy of an intermediate of the last call as a CUDA tensor (f32 or bf16)."""
        import torch
        info = TensorInfo()
        st = self.lib.outlets_get_intermediate(self.h, which, None, 0, ctypes.byref(info), None)
        if st != OK:
            self._raise(st)
        dt = torch.bfloat16 if info.dtype == BF16 else torch.float32
        out = torch.empty((info.rows, info.cols), dtype=dt, device=f"cuda:{self.device}")
        st = self.lib.outlets_get_intermediate(self.h, which, out.data_ptr(), out.numel() * out.element_size(),
                                               ctypes.byref(info), _stream_handle(stream))
        if st != OK:
            self._raise(st)
        return out


class KVCache:
    """Paged draft KV cache bound to one Predictor."""

    def __init__(self, pred: Predictor, max_slots: int, max_tokens_total: int):
        self.pred = pred
        self.lib = pred.lib
        h = c_vp()
        st = self.lib.outlets_kv_create(pred.h, max_slots, max_tokens_total, ctypes.byref(h))
        if st != OK:
            pred._raise(st)
        self.h = h

    def reset_slot(self, slot):
        st = self.lib.outlets_kv_reset_slot(self.h, slot)
        if st != OK:
            raise OutletsError(st, "bad slot")

    def truncate(self, slot, length):
        """Keep the first `length` cached positions of a slot (drop rejected draft positions)."""
        st = self.lib.outlets_kv_truncate(self.h, slot, length)
        if st != OK:
            raise OutletsError(st, "bad slot or length")

    def slot_length(self, slot):
        return self.lib.outlets_kv_slot_length(self.h, slot)

    @property
    def free_pages(self):
        return self.lib.outlets_kv_free_pages(self.h)

    def close(self):
        if getattr(self, "h", None):
            self.lib.outlets_kv_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def simulate_serving(cfg: dict, arrival, prompt_len, output_len, predicted_len):
    """Length-aware serving model of include/outlets_sched.h (host code).

    cfg keys: n_decode, max_running, route (ROUTE_RR / ROUTE_LB), order
    (ORDER_FCFS / ORDER_SJF), pf_base, pf_per_token, step_base, step_per_seq,
    step_per_kv (seconds).  Returns (finish time [n] f64, decode instance [n] i32).
    """
    lib = load()
    c = SchedConfig()
    c.n_decode, c.max_running, c.route, c.order = cfg["n_decode"], cfg["max_running"], cfg["route"], cfg["order"]
    c.pf_base_s, c.pf_per_token_s = cfg["pf_base"], cfg["pf_per_token"]
    c.step_base_s, c.step_per_seq_s, c.step_per_kv_token_s = cfg["step_base"], cfg["step_per_seq"], cfg["step_per_kv"]
    a = np.ascontiguousarray(arrival, dtype=np.float64)
    p = np.ascontiguousarray(prompt_len, dtype=np.int32)
    o = np.ascontiguousarray(output_len, dtype=np.int32)
    r = np.ascontiguousarray(predicted_len, dtype=np.float32)
    n = len(a)
    if not (len(p) == len(o) == len(r) == n):
        raise ValueError("arrays must have the same length")
    fin = np.zeros(n, np.float64)
    inst = np.zeros(n, np.int32)
    st = lib.outlets_sched_simulate(ctypes.byref(c), n, a.ctypes.data, p.ctypes.data, o.ctypes.data, r.ctypes.data,
                                    fin.ctypes.data, inst.ctypes.data)
    if st != OK:
        raise OutletsError(st, "outlets_sched_simulate rejected its arguments")
    return fin, inst
