"""HeadGuard mixed-precision KV cache for GB300 -- Python binding of the C ABI.

Thin ctypes marshalling over ``libheadguard.so`` (declared in
``include/headguard.h``): every function here has the C entry point's name,
converts its arguments (torch tensors -> device pointers, streams -> handles)
and raises :class:`HGError` on a non-zero status (and ValueError, before the
call, when a tensor argument is not a dense CUDA tensor holding the bytes the
call reads or writes through it).  All computation happens in
the library's CUDA kernels; there is no Python or CPU fallback, and importing
the compute functions without the built library raises.
"""
import ctypes
import os

from . import build as _build

__all__ = [
    "HGError", "Shape", "QuantConfig", "HeadRegions", "Cache",
    "HG_BASE_MINMAX_TOKEN", "HG_BASE_KIVI", "HG_BASE_AKVQ_HADAMARD",
    "HG_HEAD_QUANTIZED", "HG_HEAD_KEYS_ONLY", "HG_HEAD_PROTECTED",
    "hg_cache_layout", "hg_cache_create", "hg_cache_destroy", "hg_cache_head_regions",
    "hg_cache_appended", "hg_cache_reset_appended", "hg_quantize_kv", "hg_dequantize_kv",
    "hg_append_kv", "hg_decode_workspace_size", "hg_workspace_clear", "hg_workspace_status",
    "hg_check_bounded_wait", "hg_select_heads",
    "hg_decode_attention",
    "hg_decode_step", "hg_decode_attention_noalloc", "hg_cache_image_bits_per_elem",
    "hg_status_string",
    "library", "library_path",
]

HG_BASE_MINMAX_TOKEN = 0
HG_BASE_KIVI = 1
HG_BASE_AKVQ_HADAMARD = 2
HG_HEAD_QUANTIZED = 0
HG_HEAD_KEYS_ONLY = 1
HG_HEAD_PROTECTED = 2
NONE_OFFSET = (1 << 64) - 1

STATUS = {
    0: "HG_OK", 1: "HG_ERR_INVALID_ARG", 2: "HG_ERR_ALIGNMENT", 3: "HG_ERR_UNSUPPORTED",
    4: "HG_ERR_WORKSPACE_TOO_SMALL", 5: "HG_ERR_CAPACITY", 6: "HG_ERR_CUDA",
    7: "HG_ERR_ARENA_TOO_SMALL",
}


class HGError(RuntimeError):
    def __init__(self, status, where):
        self.status = status
        super().__init__("%s: %s (%s)" % (where, STATUS.get(status, status),
                                          hg_status_string(status)))


class Shape(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "batch", "num_layers", "num_kv_heads", "num_q_heads", "head_dim", "seq_len",
        "img_start", "img_len", "max_new_tokens")]


class QuantConfig(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "base", "bits", "keys_only", "kivi_group_tokens", "kivi_group_channels",
        "kivi_residual", "meta_bits", "salient_permille")]


class HeadRegions(ctypes.Structure):
    _fields_ = ([(n, ctypes.c_int32) for n in ("head_class", "nq", "bf16_prefill",
                                                "bf16_capacity")] +
                [(n, ctypes.c_uint64) for n in ("kb", "vb", "kq", "kqm", "vq", "vqm", "kimg",
                                                 "kb_bstride", "kq_bstride", "kqm_bstride",
                                                 "vq_bstride", "vqm_bstride", "kimg_bstride",
                                                 "sal", "sal_bstride")] +
                [(n, ctypes.c_int32) for n in ("n_coded", "n_salient")])


_lib = None


def library_path():
    return _build.LIB


def library():
    """Load libheadguard.so (it must have been built by build.build())."""
    global _lib
    if _lib is not None:
        return _lib
    path = _build.LIB
    if not os.path.exists(path):
        raise RuntimeError("libheadguard.so is not built (%s); run "
                           "paper_2609_35800_gb300.build.build() first" % path)
    L = ctypes.CDLL(path)
    P, i32, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_size_t
    st = ctypes.c_int
    sigs = {
        "hg_cache_layout": ([P, P, P, ctypes.POINTER(sz)], st),
        "hg_cache_create": ([P, P, P, P, sz, ctypes.POINTER(P)], st),
        "hg_cache_destroy": ([P], None),
        "hg_cache_head_regions": ([P, i32, i32, ctypes.POINTER(HeadRegions)], st),
        "hg_cache_appended": ([P, i32], i32),
        "hg_cache_reset_appended": ([P], st),
        "hg_quantize_kv": ([P, i32, i32, P, P, P], st),
        "hg_dequantize_kv": ([P, i32, i32, P, P, i32, P], st),
        "hg_append_kv": ([P, i32, i32, P, P, P], st),
        "hg_decode_workspace_size": ([P, i32, ctypes.POINTER(sz)], st),
        "hg_workspace_clear": ([P, sz, P], st),
        "hg_workspace_status": ([P, ctypes.POINTER(ctypes.c_uint32), P], st),
        "hg_check_bounded_wait": ([P, ctypes.c_uint32, P], st),
        "hg_select_heads": ([P, P, i32, i32, i32, i32, P], st),
        "hg_decode_attention": ([P, i32, i32, P, P, ctypes.c_float, P, sz, P], st),
        "hg_decode_step": ([P, i32, i32, P, P, P, P, ctypes.c_float, P, sz, P], st),
        "hg_decode_attention_noalloc": ([P, i32, i32, P, P, ctypes.c_float, P], st),
        "hg_cache_image_bits_per_elem": ([P, ctypes.POINTER(ctypes.c_double)], st),
        "hg_status_string": ([st], ctypes.c_char_p),
    }
    for name, (args, res) in sigs.items():
        f = getattr(L, name)
        f.argtypes = args
        f.restype = res
    _lib = L
    return L


def _check(status, where):
    if status != 0:
        raise HGError(status, where)


def _devs(where, *specs):
    """Addresses of device buffer arguments, each given as (x, nbytes, name).
    A torch tensor must be dense and hold at least `nbytes` bytes (the extent
    the library reads or writes through it) -- checked for every argument
    first -- and live on a CUDA device; an int is taken as a raw device
    address whose extent the caller vouches for, None as a null pointer
    (which the library rejects)."""
    for x, nbytes, name in specs:
        if x is None or isinstance(x, int):
            continue
        if not x.is_contiguous():
            raise ValueError("%s: %s must be contiguous" % (where, name))
        have = x.numel() * x.element_size()
        if have < nbytes:
            raise ValueError("%s: %s holds %d bytes, the call touches %d"
                             % (where, name, have, nbytes))
    for x, _, name in specs:
        if x is not None and not isinstance(x, int) and not x.is_cuda:
            raise ValueError("%s: %s must be a CUDA tensor" % (where, name))
    return [x if (x is None or isinstance(x, int)) else x.data_ptr() for x, _, _ in specs]


def _extent(cache, *dims, elem=2):
    """Bytes of a dense [dims...][head_dim] array of `elem`-byte entries."""
    n = elem * cache.shape.head_dim
    for d in dims:
        n *= max(int(d), 0)
    return n


def _stream(stream):
    """cudaStream_t handle: a torch.cuda.Stream, an int, or None (current torch stream)."""
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _mask_bytes(mask):
    import numpy as np
    m = np.ascontiguousarray(np.asarray(mask, dtype=np.uint8))
    return m, m.ctypes.data_as(ctypes.c_void_p)


class Cache:
    """Owning handle of an hg_cache descriptor (the arena stays caller-owned)."""

    def __init__(self, handle, arena, shape, config, mask):
        self.handle = handle
        self.arena = arena
        self.shape = shape
        self.config = config
        self.mask = mask

    def __del__(self):
        if getattr(self, "handle", None) and _lib is not None:
            _lib.hg_cache_destroy(self.handle)
            self.handle = None


def hg_status_string(status):
    return library().hg_status_string(int(status)).decode()


def hg_cache_layout(shape, config, head_mask):
    m, mp = _mask_bytes(head_mask)
    out = ctypes.c_size_t(0)
    _check(library().hg_cache_layout(ctypes.byref(shape), ctypes.byref(config), mp,
                                     ctypes.byref(out)), "hg_cache_layout")
    return out.value


def hg_cache_create(shape, config, head_mask, arena, arena_bytes=None):
    """Create the descriptor of a cache stored in `arena` (a device tensor or address)."""
    m, mp = _mask_bytes(head_mask)
    if arena_bytes is None:
        arena_bytes = arena.numel() * arena.element_size()
    h = ctypes.c_void_p()
    ap, = _devs("hg_cache_create", (arena, arena_bytes, "arena"))
    _check(library().hg_cache_create(ctypes.byref(shape), ctypes.byref(config), mp, ap,
                                     arena_bytes, ctypes.byref(h)), "hg_cache_create")
    return Cache(h, arena, shape, config, m.copy())


def hg_cache_destroy(cache):
    if cache.handle:
        library().hg_cache_destroy(cache.handle)
        cache.handle = None


def hg_cache_head_regions(cache, layer, head):
    out = HeadRegions()
    _check(library().hg_cache_head_regions(cache.handle, layer, head, ctypes.byref(out)),
           "hg_cache_head_regions")
    return out


def hg_cache_appended(cache, layer):
    return library().hg_cache_appended(cache.handle, layer)


def hg_cache_reset_appended(cache):
    _check(library().hg_cache_reset_appended(cache.handle), "hg_cache_reset_appended")


def hg_quantize_kv(cache, layer_begin, k_list, v_list, stream=None):
    n = len(k_list)
    if len(v_list) != n:
        raise ValueError("hg_quantize_kv: %d key and %d value tensors" % (n, len(v_list)))
    sh = cache.shape
    need = _extent(cache, sh.batch, sh.num_kv_heads, sh.seq_len)
    ptrs = _devs("hg_quantize_kv", *([(k, need, "k[%d]" % i) for i, k in enumerate(k_list)] +
                                     [(v, need, "v[%d]" % i) for i, v in enumerate(v_list)]))
    karr = (ctypes.c_void_p * n)(*ptrs[:n])
    varr = (ctypes.c_void_p * n)(*ptrs[n:])
    _check(library().hg_quantize_kv(cache.handle, layer_begin, n, karr, varr, _stream(stream)),
           "hg_quantize_kv")


def hg_dequantize_kv(cache, layer_begin, layer_count, k_out, v_out, out_fp32, stream=None):
    """Reconstruct layers [layer_begin, +layer_count) into k_out / v_out
    [layer_count][B][H_kv][T + appended][128] (fp32 or BF16)."""
    sh = cache.shape
    t = sh.seq_len + max(hg_cache_appended(cache, layer_begin), 0)
    need = _extent(cache, layer_count, sh.batch, sh.num_kv_heads, t, elem=4 if out_fp32 else 2)
    kp, vp = _devs("hg_dequantize_kv", (k_out, need, "k_out"), (v_out, need, "v_out"))
    _check(library().hg_dequantize_kv(cache.handle, layer_begin, layer_count, kp, vp,
                                      1 if out_fp32 else 0, _stream(stream)), "hg_dequantize_kv")


def hg_append_kv(cache, layer_begin, layer_count, k_new, v_new, stream=None):
    sh = cache.shape
    need = _extent(cache, layer_count, sh.batch, sh.num_kv_heads)
    kp, vp = _devs("hg_append_kv", (k_new, need, "k_new"), (v_new, need, "v_new"))
    _check(library().hg_append_kv(cache.handle, layer_begin, layer_count, kp, vp,
                                  _stream(stream)), "hg_append_kv")


def hg_decode_workspace_size(cache, layer_count):
    out = ctypes.c_size_t(0)
    _check(library().hg_decode_workspace_size(cache.handle, layer_count, ctypes.byref(out)),
           "hg_decode_workspace_size")
    return out.value


def hg_workspace_clear(workspace, nbytes=None, stream=None):
    """Zero a decode workspace; workspace None clears the status word of the
    allocation-free entry point's scratch on the current device."""
    if workspace is None:
        nbytes = 0
    elif nbytes is None:
        nbytes = workspace.numel() * workspace.element_size()
    wp, = _devs("hg_workspace_clear", (workspace, nbytes, "workspace"))
    _check(library().hg_workspace_clear(wp, nbytes, _stream(stream)), "hg_workspace_clear")


def hg_workspace_status(workspace, stream=None):
    """Status word of a decode workspace (waits for the stream); 0 = healthy.
    workspace None: the status word of the allocation-free entry point's scratch
    on the current device."""
    out = ctypes.c_uint32(0)
    wp, = _devs("hg_workspace_status", (workspace, 4, "workspace"))
    _check(library().hg_workspace_status(wp, ctypes.byref(out), _stream(stream)),
           "hg_workspace_status")
    return out.value


def hg_check_bounded_wait(word, rounds, stream=None):
    """Run the bounded-wait self-check into the device word `word` (see the header)."""
    wp, = _devs("hg_check_bounded_wait", (word, 4, "word"))
    _check(library().hg_check_bounded_wait(wp, int(rounds), _stream(stream)),
           "hg_check_bounded_wait")


def hg_select_heads(g_scores, o_scores, num_layers, num_q_heads, num_kv_heads, k=-1):
    """Protected-head mask (numpy uint8 [num_layers][num_kv_heads]) from host
    per-query-head scores [num_layers][num_q_heads] (see the header)."""
    import numpy as np
    g = np.ascontiguousarray(np.asarray(g_scores, dtype=np.float32))
    o = np.ascontiguousarray(np.asarray(o_scores, dtype=np.float32))
    mask = np.zeros((num_layers, num_kv_heads), dtype=np.uint8)
    _check(library().hg_select_heads(g.ctypes.data_as(ctypes.c_void_p), o.ctypes.data_as(ctypes.c_void_p),
                                     num_layers, num_q_heads, num_kv_heads, int(k),
                                     mask.ctypes.data_as(ctypes.c_void_p)), "hg_select_heads")
    return mask


def hg_decode_attention(cache, layer_begin, layer_count, q, out, softmax_scale, workspace,
                        workspace_bytes=None, stream=None):
    if workspace_bytes is None:
        workspace_bytes = workspace.numel() * workspace.element_size()
    sh = cache.shape
    need = _extent(cache, layer_count, sh.batch, sh.num_q_heads)
    qp, op, wp = _devs("hg_decode_attention", (q, need, "q"), (out, need, "out"),
                       (workspace, workspace_bytes, "workspace"))
    _check(library().hg_decode_attention(cache.handle, layer_begin, layer_count, qp, op,
                                         float(softmax_scale), wp, workspace_bytes,
                                         _stream(stream)), "hg_decode_attention")


def hg_decode_step(cache, layer_begin, layer_count, q, k_new, v_new, out, softmax_scale, workspace,
                   workspace_bytes=None, stream=None):
    """Append the step's K/V and run decode attention including it, in one launch."""
    if workspace_bytes is None:
        workspace_bytes = workspace.numel() * workspace.element_size()
    sh = cache.shape
    nq = _extent(cache, layer_count, sh.batch, sh.num_q_heads)
    nkv = _extent(cache, layer_count, sh.batch, sh.num_kv_heads)
    qp, kp, vp, op, wp = _devs("hg_decode_step", (q, nq, "q"), (k_new, nkv, "k_new"),
                               (v_new, nkv, "v_new"), (out, nq, "out"),
                               (workspace, workspace_bytes, "workspace"))
    _check(library().hg_decode_step(cache.handle, layer_begin, layer_count, qp, kp, vp, op,
                                    float(softmax_scale), wp, workspace_bytes, _stream(stream)),
           "hg_decode_step")


def hg_decode_attention_noalloc(cache, layer_begin, layer_count, q, out, softmax_scale,
                                stream=None):
    """Decode attention with the library's static 32 MiB scratch as workspace (no allocation)."""
    sh = cache.shape
    need = _extent(cache, layer_count, sh.batch, sh.num_q_heads)
    qp, op = _devs("hg_decode_attention_noalloc", (q, need, "q"), (out, need, "out"))
    _check(library().hg_decode_attention_noalloc(cache.handle, layer_begin, layer_count, qp, op,
                                                 float(softmax_scale), _stream(stream)),
           "hg_decode_attention_noalloc")


def hg_cache_image_bits_per_elem(cache):
    out = ctypes.c_double(0)
    _check(library().hg_cache_image_bits_per_elem(cache.handle, ctypes.byref(out)),
           "hg_cache_image_bits_per_elem")
    return out.value
