"""Python binding of libdas.so, the GB300 library for the data-parallel hot path
of DAS-Wave decoding ("Shallow Queries, Mature Values: Depth-Asynchronous
Self-Speculation for Looped Transformers").

Argument marshalling only: every computation runs in the library's CUDA
kernels.  PyTorch provides device memory and streams.  The names match the C
ABI in include/das.h:

    das_workspace_size      bytes of scratch the attention calls need
    das_mature_v_attention  Eqs. 2-3 with explicit read depths (Eq. 4)
    das_verify_attention    full-depth verify attention (Sec. 3.4, Eq. 7)
    das_greedy_accept       greedy acceptance (Sec. 3.4)
    das_kv_append           commit of accepted K/V at every depth (App. B.1)
    das_wave_readout        DAS-Wave shifted token readout (Eq. 6)
    DepthKVCacheF8, das_mature_v_attention_f8, das_kv_append_f8
                            the cache variant with depths below R stored as
                            e4m3 (not in the paper)
    AttentionCall           the attention calls with arguments checked once, for
                            loops that call with the same tensors every step
    wave_widths, WaveRefinement
                            DAS-Wave's round schedule (Eq. 5) and the device
                            side of its carried parallel refinement (Sec. 3.3)

If libdas.so is missing the import fails: there is no fallback.
"""
import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libdas.so")

DAS_OK, DAS_ERR_INVALID_ARG, DAS_ERR_UNSUPPORTED, DAS_ERR_WORKSPACE, DAS_ERR_CUDA = range(5)


class DasError(RuntimeError):
    def __init__(self, code, what):
        super().__init__(f"{what}: {status_string(code)} (status {code})")
        self.code = code


class das_kv_cache(ctypes.Structure):
    _fields_ = [("k", ctypes.c_void_p), ("v", ctypes.c_void_p), ("depths", ctypes.c_int),
                ("layers", ctypes.c_int), ("batch", ctypes.c_int), ("capacity", ctypes.c_int),
                ("kv_heads", ctypes.c_int), ("head_dim", ctypes.c_int)]


class das_kv_cache_f8(ctypes.Structure):
    _fields_ = [("k_top", ctypes.c_void_p), ("v_top", ctypes.c_void_p),
                ("k_low", ctypes.c_void_p), ("v_low", ctypes.c_void_p), ("depths", ctypes.c_int),
                ("layers", ctypes.c_int), ("batch", ctypes.c_int), ("capacity", ctypes.c_int),
                ("kv_heads", ctypes.c_int), ("head_dim", ctypes.c_int)]


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is not built: run `python -m paper_2609_34538_gb300.build` "
                          "(needs nvcc with sm_103a support)")
    lib = ctypes.CDLL(LIB_PATH)
    i, p, f, sz = ctypes.c_int, ctypes.c_void_p, ctypes.c_float, ctypes.c_size_t
    cp = ctypes.POINTER(das_kv_cache)
    lib.das_workspace_size.argtypes = [cp, i, i]
    lib.das_workspace_size.restype = sz
    lib.das_mature_v_attention.argtypes = [cp, i, i, i, p, p, i, p, p, p, i, f, p, p, p, sz, p]
    lib.das_mature_v_attention.restype = i
    lib.das_verify_attention.argtypes = [cp, i, i, p, p, i, p, p, p, i, f, p, p, p, sz, p]
    lib.das_verify_attention.restype = i
    lib.das_greedy_accept.argtypes = [p, p, i, i, i, p, p, p, p]
    lib.das_greedy_accept.restype = i
    lib.das_kv_append.argtypes = [cp, p, p, p, i, p, p, p]
    lib.das_kv_append.restype = i
    lib.das_wave_readout.argtypes = [p, i, i, i, p, i, p]
    lib.das_wave_readout.restype = i
    cp8 = ctypes.POINTER(das_kv_cache_f8)
    lib.das_workspace_size_f8.argtypes = [cp8, i, i]
    lib.das_workspace_size_f8.restype = sz
    lib.das_mature_v_attention_f8.argtypes = [cp8, i, i, i, p, p, i, p, p, p, i, f, p, p, p, sz, p]
    lib.das_mature_v_attention_f8.restype = i
    lib.das_kv_append_f8.argtypes = [cp8, p, p, p, i, p, p, p]
    lib.das_kv_append_f8.restype = i
    lib.das_mature_v_attention_noalloc.argtypes = [cp, i, i, i, p, p, i, p, p, p, i, f, p, p, p]
    lib.das_mature_v_attention_noalloc.restype = i
    lib.das_noalloc_status.argtypes = [p, p]
    lib.das_noalloc_status.restype = i
    lib.das_status_string.argtypes = [i]
    lib.das_status_string.restype = ctypes.c_char_p
    return lib


LIB = _load()


def status_string(code):
    return LIB.das_status_string(int(code)).decode()


def _check(code, what):
    if code != DAS_OK:
        raise DasError(code, what)


def _stream(stream):
    s = torch.cuda.current_stream() if stream is None else stream
    return s.cuda_stream


def _ptr(t):
    return t.data_ptr() if t is not None else 0


def _need(t, dtype, name, ndim=None):
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_cuda:
        raise ValueError(f"{name} must be on a CUDA device")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if ndim is not None and t.dim() != ndim:
        raise ValueError(f"{name} must have {ndim} dims, got {tuple(t.shape)}")


class DepthKVCache:
    """A depth-indexed cache: k, v bf16 [depths][layers][batch][capacity][kv_heads][head_dim]."""

    def __init__(self, k, v):
        _need(k, torch.bfloat16, "k", 6)
        _need(v, torch.bfloat16, "v", 6)
        if k.shape != v.shape:
            raise ValueError("k and v shapes differ")
        self.k, self.v = k, v
        R, L, B, cap, H, D = k.shape
        self.desc = das_kv_cache(k.data_ptr(), v.data_ptr(), R, L, B, cap, H, D)

    @classmethod
    def empty(cls, depths, layers, batch, capacity, kv_heads, head_dim, device="cuda"):
        shape = (depths, layers, batch, capacity, kv_heads, head_dim)
        return cls(torch.empty(shape, dtype=torch.bfloat16, device=device),
                   torch.empty(shape, dtype=torch.bfloat16, device=device))

    @property
    def shape(self):
        return tuple(self.k.shape)


def das_workspace_size(cache, num_q_heads, max_block):
    return int(LIB.das_workspace_size(ctypes.byref(cache.desc), num_q_heads, max_block))


def new_workspace(cache, num_q_heads, max_block, device=None):
    """Zeroed workspace tensor (uint8) of the size the attention calls need."""
    n = das_workspace_size(cache, num_q_heads, max_block)
    if n == 0:
        raise DasError(DAS_ERR_UNSUPPORTED, "das_workspace_size")
    return torch.zeros(n, dtype=torch.uint8, device=device or cache.k.device)


def workspace_status(workspace):
    """The workspace status word (bit 0: an internal wait timed out; bit 1: a
    prefix or block length was out of range and clamped).  Synchronises."""
    return int(workspace[:4].view(torch.int32).item())


def _attention_shapes(cache, prefix_len, block_len, q, k_blk, v_blk, out, lse):
    """Checks every tensor of an attention call against the cache's shape
    (allocating out / lse when omitted); returns (max_block, Hq, out, lse).
    Raises before anything is launched."""
    _need(prefix_len, torch.int32, "prefix_len", 1)
    _need(block_len, torch.int32, "block_len", 1)
    _need(q, torch.bfloat16, "q", 4)
    _need(k_blk, torch.bfloat16, "k_blk", 4)
    _need(v_blk, torch.bfloat16, "v_blk", 4)
    R, L, B, cap, H, D = cache.shape
    Bq, T, Hq, Dq = q.shape
    if Bq != B or Dq != D or prefix_len.numel() != B or block_len.numel() != B:
        raise ValueError("q / length shapes do not match the cache")
    if tuple(k_blk.shape) != (B, T, H, D) or tuple(v_blk.shape) != (B, T, H, D):
        raise ValueError("k_blk / v_blk must be [batch][max_block][kv_heads][head_dim]")
    if out is None:
        out = torch.empty_like(q)
    if lse is None:
        lse = torch.empty((B, Hq, T), dtype=torch.float32, device=q.device)
    _need(out, torch.bfloat16, "out", 4)
    _need(lse, torch.float32, "lse", 3)
    if tuple(out.shape) != tuple(q.shape) or tuple(lse.shape) != (B, Hq, T):
        raise ValueError("out must be like q and lse [batch][num_q_heads][max_block]")
    return T, Hq, out, lse


def _attention_args(cache, prefix_len, block_len, q, k_blk, v_blk, out, lse, workspace):
    T, Hq, out, lse = _attention_shapes(cache, prefix_len, block_len, q, k_blk, v_blk, out, lse)
    _need(workspace, torch.uint8, "workspace", 1)
    return T, Hq, out, lse


def das_mature_v_attention(cache, layer, key_depth, value_depth, prefix_len, block_len, q, k_blk,
                           v_blk, workspace, out=None, lse=None, softmax_scale=0.0, stream=None):
    """Depth-asynchronous attention (Eqs. 2-3); returns (out, lse)."""
    T, Hq, out, lse = _attention_args(cache, prefix_len, block_len, q, k_blk, v_blk, out, lse,
                                      workspace)
    _check(LIB.das_mature_v_attention(
        ctypes.byref(cache.desc), layer, key_depth, value_depth, _ptr(prefix_len),
        _ptr(block_len), T, _ptr(q), _ptr(k_blk), _ptr(v_blk), Hq, float(softmax_scale),
        _ptr(out), _ptr(lse), _ptr(workspace), workspace.numel(), _stream(stream)),
        "das_mature_v_attention")
    return out, lse


def das_mature_v_attention_noalloc(cache, layer, key_depth, value_depth, prefix_len, block_len, q,
                                   k_blk, v_blk, out=None, lse=None, softmax_scale=0.0,
                                   stream=None):
    """das_mature_v_attention for callers that cannot allocate device memory:
    the split-K scratch is a fixed array inside the library (shared by every
    call on a device; calls that overlap on the GPU race).  `out` and `lse`
    must be given by such callers; they are allocated here only for
    convenience when omitted.  Shapes are checked as for the workspace entry
    point, before anything is launched."""
    T, Hq, out, lse = _attention_shapes(cache, prefix_len, block_len, q, k_blk, v_blk, out, lse)
    _check(LIB.das_mature_v_attention_noalloc(
        ctypes.byref(cache.desc), layer, key_depth, value_depth, _ptr(prefix_len),
        _ptr(block_len), T, _ptr(q), _ptr(k_blk), _ptr(v_blk), Hq, float(softmax_scale),
        _ptr(out), _ptr(lse), _stream(stream)), "das_mature_v_attention_noalloc")
    return out, lse


def noalloc_status(stream=None):
    """The status word of the last das_mature_v_attention_noalloc call on the
    current device (bits as workspace_status).  Synchronises the stream."""
    host = torch.zeros(1, dtype=torch.int32)
    s = torch.cuda.current_stream() if stream is None else stream
    _check(LIB.das_noalloc_status(host.data_ptr(), s.cuda_stream), "das_noalloc_status")
    s.synchronize()
    return int(host.item())


def das_verify_attention(cache, layer, depth, prefix_len, block_len, q, k_blk, v_blk, workspace,
                         out=None, lse=None, softmax_scale=0.0, stream=None):
    """Full-depth verify attention (Sec. 3.4); returns (out, lse)."""
    T, Hq, out, lse = _attention_args(cache, prefix_len, block_len, q, k_blk, v_blk, out, lse,
                                      workspace)
    _check(LIB.das_verify_attention(
        ctypes.byref(cache.desc), layer, depth, _ptr(prefix_len), _ptr(block_len), T, _ptr(q),
        _ptr(k_blk), _ptr(v_blk), Hq, float(softmax_scale), _ptr(out), _ptr(lse),
        _ptr(workspace), workspace.numel(), _stream(stream)), "das_verify_attention")
    return out, lse


class AttentionCall:
    """Attention calls with fixed arguments, checked once.

    A serving loop calls attention with the same cache, lengths, inputs,
    outputs and workspace every step.  This object checks them when it is
    built and keeps their marshalled pointers, so each call below is a single
    C call.  The tensors must stay alive, in place and unchanged in shape
    while the object is used (their contents may change between calls).

        call = AttentionCall(cache, prefix_len, block_len, q, k_blk, v_blk, ws)
        out, lse = call.mature_v(layer, key_depth, value_depth, stream)
        out, lse = call.verify(layer, depth, stream)
    """

    def __init__(self, cache, prefix_len, block_len, q, k_blk, v_blk, workspace, out=None,
                 lse=None, softmax_scale=0.0):
        T, Hq, out, lse = _attention_args(cache, prefix_len, block_len, q, k_blk, v_blk, out,
                                          lse, workspace)
        self.cache, self.out, self.lse = cache, out, lse
        self._keep = (prefix_len, block_len, q, k_blk, v_blk, workspace)
        self._desc = ctypes.byref(cache.desc)
        self._args = (_ptr(prefix_len), _ptr(block_len), T, _ptr(q), _ptr(k_blk), _ptr(v_blk),
                      Hq, float(softmax_scale), _ptr(out), _ptr(lse), _ptr(workspace),
                      workspace.numel())

    def mature_v(self, layer, key_depth, value_depth, stream=None):
        """das_mature_v_attention (Eqs. 2-3) with this object's arguments."""
        _check(LIB.das_mature_v_attention(self._desc, layer, key_depth, value_depth, *self._args,
                                          _stream(stream)), "das_mature_v_attention")
        return self.out, self.lse

    def verify(self, layer, depth, stream=None):
        """das_verify_attention (Sec. 3.4) with this object's arguments."""
        _check(LIB.das_verify_attention(self._desc, layer, depth, *self._args, _stream(stream)),
               "das_verify_attention")
        return self.out, self.lse


def das_greedy_accept(logits, draft_ids, accepted=None, target_ids=None, next_token=None,
                      stream=None):
    """Greedy acceptance (Sec. 3.4); returns (accepted, target_ids, next_token)."""
    _need(logits, torch.float32, "logits", 3)
    _need(draft_ids, torch.int32, "draft_ids", 2)
    B, W, V = logits.shape
    if tuple(draft_ids.shape) != (B, W):
        raise ValueError("draft_ids must be [B][W]")
    dev = logits.device
    accepted = torch.empty(B, dtype=torch.int32, device=dev) if accepted is None else accepted
    target_ids = torch.empty((B, W), dtype=torch.int32, device=dev) if target_ids is None else target_ids
    next_token = torch.empty(B, dtype=torch.int32, device=dev) if next_token is None else next_token
    _need(accepted, torch.int32, "accepted", 1)
    _need(target_ids, torch.int32, "target_ids", 2)
    _need(next_token, torch.int32, "next_token", 1)
    _check(LIB.das_greedy_accept(_ptr(logits), _ptr(draft_ids), B, W, V, _ptr(accepted),
                                 _ptr(target_ids), _ptr(next_token), _stream(stream)),
           "das_greedy_accept")
    return accepted, target_ids, next_token


def das_kv_append(cache, k_new, v_new, accepted, prefix_len, error_flag, stream=None):
    """Commit (App. B.1): copy min(accepted+1, W) staged positions per sequence
    at every depth and layer; prefix_len grows in place."""
    _need(k_new, torch.bfloat16, "k_new", 6)
    _need(v_new, torch.bfloat16, "v_new", 6)
    _need(accepted, torch.int32, "accepted", 1)
    _need(prefix_len, torch.int32, "prefix_len", 1)
    _need(error_flag, torch.int32, "error_flag")
    R, L, B, cap, H, D = cache.shape
    W = k_new.shape[3]
    if tuple(k_new.shape) != (R, L, B, W, H, D) or k_new.shape != v_new.shape:
        raise ValueError("k_new / v_new must be [depths][layers][batch][W][kv_heads][head_dim]")
    _check(LIB.das_kv_append(ctypes.byref(cache.desc), _ptr(k_new), _ptr(v_new), _ptr(accepted),
                             W, _ptr(prefix_len), _ptr(error_flag), _stream(stream)),
           "das_kv_append")


def das_wave_readout(logits, tokens, stream=None):
    """Shifted readout of a DAS-Wave round (Eq. 6), in place:
    tokens[b][i + 1] = argmax_v logits[b][i][v] for i < W; returns tokens."""
    _need(logits, torch.float32, "logits", 3)
    _need(tokens, torch.int32, "tokens", 2)
    B, W, V = logits.shape
    if tokens.shape[0] != B or tokens.shape[1] < W + 1:
        raise ValueError("tokens must be [B][>= W + 1] for logits [B][W][vocab]")
    _check(LIB.das_wave_readout(_ptr(logits), B, W, V, _ptr(tokens), tokens.shape[1],
                                _stream(stream)), "das_wave_readout")
    return tokens


def wave_widths(gamma, w_init, rounds):
    """Active widths W_j = min(gamma, W_init + j) of rounds j = 0 .. J-1 (Eq. 5)."""
    if gamma < 1 or w_init < 1 or w_init > gamma or rounds < 0:
        raise ValueError("need 1 <= W_init <= gamma and J >= 0")
    return [min(gamma, w_init + j) for j in range(rounds)]


class WaveRefinement:
    """The device side of DAS-Wave's carried parallel refinement (Sec. 3.3).

    Round j works on the W_j = min(gamma, W_init + j) active positions
    [x_t, z_1 .. z_{W_j - 1}] (Eq. 5): k recurrent draft updates, each running
    the L core layers, whose attention reads the verified prefix at Deep K/V
    (key and value depth R) and the active positions' own K/V under the
    causal mask; then the shifted readout (Eq. 6) revises the token guesses
    and the last position's readout becomes the candidate that enters the
    window next round.  Token guesses start as the repeated anchor.

    The looped model between the attention calls is the caller's:
      step(j, s, layer) -> (q, k_blk, v_blk, out, lse) buffers of the call
          (q/out [B][gamma][Hq][D], k_blk/v_blk [B][gamma][Hkv][D],
          lse [B][Hq][gamma]; rows >= W_j are inactive),
      logits(j) -> fp32 [B][W_j][vocab] readout logits of round j.
    After run(), tokens[:, :w] is the verifier input [x_t, y_1 .. y_{w-1}] and
    tokens[:, w] the final readout y_w, w = W_{J-1}.
    """

    def __init__(self, cache, prefix_len, workspace, num_q_heads, gamma=32, w_init=2, rounds=24,
                 k_steps=2):
        R, L, B, cap, H, D = cache.shape
        self.cache, self.prefix_len, self.workspace = cache, prefix_len, workspace
        self.num_q_heads, self.gamma, self.k_steps, self.layers = num_q_heads, gamma, k_steps, L
        self.widths = wave_widths(gamma, w_init, rounds)
        dev = cache.k.device
        # block_len of every distinct width, made once
        self._bl = {w: torch.full((B,), w, dtype=torch.int32, device=dev)
                    for w in sorted(set(self.widths))}
        self.tokens = torch.zeros((B, gamma + 1), dtype=torch.int32, device=dev)

    def run(self, anchor, step, logits, stream=None):
        """anchor: device int32 [B].  Returns the token buffer [B][gamma + 1]."""
        R = self.cache.shape[0]
        s_ = torch.cuda.current_stream() if stream is None else stream
        with torch.cuda.stream(s_):
            self.tokens.copy_(anchor.view(-1, 1).expand_as(self.tokens))
        for j, W in enumerate(self.widths):
            for s in range(self.k_steps):
                for layer in range(self.layers):
                    q, kb, vb, out, lse = step(j, s, layer)
                    das_mature_v_attention(self.cache, layer, R, R, self.prefix_len,
                                           self._bl[W], q, kb, vb, self.workspace, out=out,
                                           lse=lse, stream=s_)
            das_wave_readout(logits(j), self.tokens, stream=s_)
        return self.tokens


class DepthKVCacheF8:
    """A depth-indexed cache with depth R in bf16 (k_top, v_top
    [layers][batch][capacity][kv_heads][head_dim]) and depths 1..R-1 as e4m3
    codes (k_low, v_low uint8 [depths-1][layers][batch][capacity][kv_heads][head_dim])."""

    def __init__(self, k_top, v_top, k_low=None, v_low=None):
        _need(k_top, torch.bfloat16, "k_top", 5)
        _need(v_top, torch.bfloat16, "v_top", 5)
        if k_top.shape != v_top.shape:
            raise ValueError("k_top and v_top shapes differ")
        L, B, cap, H, D = k_top.shape
        R = 1
        if k_low is not None or v_low is not None:
            _need(k_low, torch.uint8, "k_low", 6)
            _need(v_low, torch.uint8, "v_low", 6)
            if k_low.shape != v_low.shape or tuple(k_low.shape[1:]) != tuple(k_top.shape):
                raise ValueError("k_low / v_low must be [depths-1] + k_top.shape")
            R = k_low.shape[0] + 1
        self.k_top, self.v_top, self.k_low, self.v_low = k_top, v_top, k_low, v_low
        self.desc = das_kv_cache_f8(k_top.data_ptr(), v_top.data_ptr(), _ptr(k_low), _ptr(v_low),
                                    R, L, B, cap, H, D)

    @classmethod
    def empty(cls, depths, layers, batch, capacity, kv_heads, head_dim, device="cuda"):
        top = (layers, batch, capacity, kv_heads, head_dim)
        low = (depths - 1,) + top
        mk = lambda shape, dt: torch.empty(shape, dtype=dt, device=device)
        return cls(mk(top, torch.bfloat16), mk(top, torch.bfloat16),
                   mk(low, torch.uint8) if depths > 1 else None,
                   mk(low, torch.uint8) if depths > 1 else None)

    @property
    def shape(self):
        d = self.desc
        return (d.depths, d.layers, d.batch, d.capacity, d.kv_heads, d.head_dim)


def new_workspace_f8(cache, num_q_heads, max_block, device=None):
    n = int(LIB.das_workspace_size_f8(ctypes.byref(cache.desc), num_q_heads, max_block))
    if n == 0:
        raise DasError(DAS_ERR_UNSUPPORTED, "das_workspace_size_f8")
    return torch.zeros(n, dtype=torch.uint8, device=device or cache.k_top.device)


def das_mature_v_attention_f8(cache, layer, key_depth, value_depth, prefix_len, block_len, q,
                              k_blk, v_blk, workspace, out=None, lse=None, softmax_scale=0.0,
                              stream=None):
    """das_mature_v_attention on an e4m3 cache (DepthKVCacheF8); returns (out, lse)."""
    T, Hq, out, lse = _attention_args(cache, prefix_len, block_len, q, k_blk, v_blk, out, lse,
                                      workspace)
    _check(LIB.das_mature_v_attention_f8(
        ctypes.byref(cache.desc), layer, key_depth, value_depth, _ptr(prefix_len),
        _ptr(block_len), T, _ptr(q), _ptr(k_blk), _ptr(v_blk), Hq, float(softmax_scale),
        _ptr(out), _ptr(lse), _ptr(workspace), workspace.numel(), _stream(stream)),
        "das_mature_v_attention_f8")
    return out, lse


def das_kv_append_f8(cache, k_new, v_new, accepted, prefix_len, error_flag, stream=None):
    """The commit into an e4m3 cache: depth R copied, depths below R rounded to
    e4m3 (nearest, ties to even, saturating at +-448)."""
    _need(k_new, torch.bfloat16, "k_new", 6)
    _need(v_new, torch.bfloat16, "v_new", 6)
    _need(accepted, torch.int32, "accepted", 1)
    _need(prefix_len, torch.int32, "prefix_len", 1)
    _need(error_flag, torch.int32, "error_flag")
    R, L, B, cap, H, D = cache.shape
    W = k_new.shape[3]
    if tuple(k_new.shape) != (R, L, B, W, H, D) or k_new.shape != v_new.shape:
        raise ValueError("k_new / v_new must be [depths][layers][batch][W][kv_heads][head_dim]")
    _check(LIB.das_kv_append_f8(ctypes.byref(cache.desc), _ptr(k_new), _ptr(v_new),
                                _ptr(accepted), W, _ptr(prefix_len), _ptr(error_flag),
                                _stream(stream)), "das_kv_append_f8")
