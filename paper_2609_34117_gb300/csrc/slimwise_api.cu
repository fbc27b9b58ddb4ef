// slimwise_api.cu -- the C ABI declared in include/slimwise_moe.h: argument
// checks, workspace layout, TMA descriptors, and the four launches of one
// decode MoE layer (route/top-k -> group/gather -> expert FFN -> combine).
#include <algorithm>
#include <cmath>
#include <cstring>
#include <mutex>

#include <cudaTypedefs.h>

#include "common.cuh"

using namespace slimwise;

namespace {

struct DeviceInfo {
  int sms = 0;
  int smem_optin = 0;
  bool ready = false;
};

std::mutex g_mu;
DeviceInfo g_dev[64];
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

int device_info(DeviceInfo *out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64)
    return SLIMWISE_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_mu);
  DeviceInfo &di = g_dev[dev];
  if (!di.ready) {
    if (cudaDeviceGetAttribute(&di.sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&di.smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) !=
            cudaSuccess)
      return SLIMWISE_ERR_CUDA;
    di.ready = true;
  }
  if (!g_encode) {
    void *fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                         cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !fn)
      return SLIMWISE_ERR_CUDA;
    g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  }
  *out = di;
  return SLIMWISE_OK;
}

// 2-D bf16 tensor map: `rows` x `cols` row-major, box `box_rows` x 64,
// 128-byte swizzle, zero fill outside the tensor.
int encode_map(CUtensorMap *map, const void *base, uint64_t rows, uint64_t cols,
               uint32_t box_rows) {
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {(cuuint32_t)kBlockK, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                        const_cast<void *>(base), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? SLIMWISE_OK : SLIMWISE_ERR_CUDA;
}

bool aligned(const void *p, uintptr_t a) {
  return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0;
}

int check_shape(const slimwise_moe_shape *s, int32_t top_k, int32_t m_ret) {
  if (!s) return SLIMWISE_ERR_INVALID_ARG;
  if (s->num_tokens < 0 || s->num_tokens > (1 << 20)) return SLIMWISE_ERR_INVALID_ARG;
  // a routing CTA stages at least one fp32 hidden row in shared memory
  if (s->hidden < 128 || s->hidden % 128 != 0 || s->hidden > 32768)
    return SLIMWISE_ERR_UNSUPPORTED_SHAPE;
  if (s->inter < 64 || s->inter % 64 != 0 || s->inter > 65536)
    return SLIMWISE_ERR_UNSUPPORTED_SHAPE;
  if (s->num_experts < 1 || s->num_experts > kMaxExperts)
    return SLIMWISE_ERR_UNSUPPORTED_SHAPE;
  if (m_ret < 1 || m_ret > s->num_experts) return SLIMWISE_ERR_INVALID_ARG;
  if (top_k < 1 || top_k > kMaxTopK || top_k > m_ret) return SLIMWISE_ERR_INVALID_ARG;
  if ((uint64_t)s->num_experts * 2 * s->inter > 0xFFFFFFFFull ||
      (uint64_t)s->num_experts * s->hidden > 0xFFFFFFFFull)
    return SLIMWISE_ERR_UNSUPPORTED_SHAPE;
  return SLIMWISE_OK;
}

Dims make_dims(const slimwise_moe_shape *s, int32_t top_k, int32_t m_ret, int32_t Is = 0) {
  Dims d;
  d.B = s->num_tokens;
  d.H = s->hidden;
  d.E = s->num_experts;
  d.I = s->inter;
  d.k = top_k;
  d.m_ret = m_ret;
  d.tok_chunk = token_chunk_for(d.B, top_k, m_ret);
  if (Is > 0) {
    // the shared expert takes every token: at least 64 of them per entry, so
    // its weight tiles pass through the SMs B/64 times rather than B/16
    // (a larger token slot per stage, a few stages fewer for the routed items)
    const int want = pow2_at_least(d.B) < 64 ? pow2_at_least(d.B) : 64;
    if (d.tok_chunk < want) d.tok_chunk = want;
  }
  d.Is = Is;
  d.S = Is > 0 ? (d.B + d.tok_chunk - 1) / d.tok_chunk : 0;
  d.wide = (Is == 0 && d.I % (2 * kGateRows) == 0 && d.H % (2 * kTileRows) == 0 &&
            d.tok_chunk >= kWideMinChunk && d.tok_chunk <= kWideMaxChunk &&
            m_ret >= kWideMinPool) ? 1 : 0;
  d.pair = 0;  // CTA-pair items only on request (apply_item_form)
  return d;
}

// The caller's choice of work-item form (slimwise_decode_opts.ffn_items).
void apply_item_form(Dims *d, int32_t form) {
  const bool can_pair = d->Is == 0 && d->I % (2 * kGateRows) == 0 && d->H % (2 * kTileRows) == 0;
  if (form > 0 && can_pair) {
    d->pair = 1;
    d->wide = 0;
  } else if (form < 0) {
    d->pair = 0;
  }
}

int check_workspace(const slimwise_moe_shape *s, int32_t top_k, void *ws,
                    size_t ws_bytes, WsLayout *L, int32_t Is = 0) {
  if (!ws) return SLIMWISE_ERR_INVALID_ARG;
  if (!aligned(ws, 256)) return SLIMWISE_ERR_UNSUPPORTED_SHAPE;
  *L = make_layout(s->num_tokens, s->hidden, s->num_experts, s->inter, top_k, Is);
  return ws_bytes >= L->total ? SLIMWISE_OK : SLIMWISE_ERR_WORKSPACE;
}

int copy_out(void *dst, const void *src, size_t bytes, cudaStream_t st) {
  if (!dst || !bytes) return SLIMWISE_OK;
  return cudaMemcpyAsync(dst, src, bytes, cudaMemcpyDeviceToDevice, st) == cudaSuccess
             ? SLIMWISE_OK
             : SLIMWISE_ERR_CUDA;
}

int copy_group_outputs(const Ws &w, const Dims &d, cudaStream_t st, int32_t *counts,
                       int32_t *offsets, int32_t *union_ids, int32_t *union_size,
                       int32_t *perm, int32_t *pos) {
  const size_t slots = (size_t)d.B * d.k;
  int rc = SLIMWISE_OK;
  if (!rc) rc = copy_out(counts, w.counts, (size_t)d.E * 4, st);
  if (!rc) rc = copy_out(offsets, w.offsets, (size_t)(d.E + 1) * 4, st);
  if (!rc) rc = copy_out(union_ids, w.union_ids, (size_t)d.E * 4, st);
  if (!rc) rc = copy_out(union_size, w.ctrl + kCtrlUnionSize, 4, st);
  if (!rc) rc = copy_out(perm, w.perm, slots * 4, st);
  if (!rc) rc = copy_out(pos, w.pos, slots * 4, st);
  return rc;
}

// The FFN kernel's tensor maps for one call.  Encoding them costs host time
// on every call, so the maps of the last call on this thread are kept and
// reused while the pointers and sizes they describe are unchanged.
// The shared expert of Sec. 3.3 (inter == 0: none).
struct SharedExpert {
  const float *gate;      // fp32 [H]
  const void *gate_up;    // bf16 [2 Is, H]
  const void *down;       // bf16 [H, Is]
  int32_t inter;          // Is
};

// The weight maps depend on the weight tensors only; the token maps on the
// workspace, the batch and the token chunk.  They are cached separately, so
// that rotating between weight copies re-encodes two or four maps, not the
// token maps of every box height.
struct WeightMapsKey {
  const void *w_gu, *w_down, *gu_s, *down_s;
  int E, H, I, Is, device;
  bool operator==(const WeightMapsKey &o) const {
    return w_gu == o.w_gu && w_down == o.w_down && gu_s == o.gu_s && down_s == o.down_s &&
           E == o.E && H == o.H && I == o.I && Is == o.Is && device == o.device;
  }
};
struct TokenMapsKey {
  const void *xp, *act, *xt, *act_s;
  int H, I, Is, B, tok_chunk, pair, device;
  uint64_t slots;
  bool operator==(const TokenMapsKey &o) const {
    return xp == o.xp && act == o.act && xt == o.xt && act_s == o.act_s && H == o.H &&
           I == o.I && Is == o.Is && B == o.B && tok_chunk == o.tok_chunk && pair == o.pair &&
           device == o.device && slots == o.slots;
  }
};

bool ffn_maps_for(FfnMaps *maps, const void *w_gate_up, const void *w_down, const Ws &w,
                  const Dims &d, uint64_t slots, const SharedExpert &se) {
  thread_local bool have_w = false, have_t = false;
  thread_local WeightMapsKey last_w;
  thread_local TokenMapsKey last_t;
  thread_local FfnMaps cached;  // both halves of the last call on this thread
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  const WeightMapsKey kw = {w_gate_up, w_down, se.gate_up, se.down, d.E, d.H, d.I, d.Is, dev};
  const TokenMapsKey kt = {w.xp, w.act, w.xt, w.act_s, d.H, d.I, d.Is, d.B, d.tok_chunk, d.pair,
                          dev, slots};
  if (!(have_w && kw == last_w)) {
    have_w = false;
    if (encode_map(&cached.w_gu, w_gate_up, (uint64_t)d.E * 2 * d.I, d.H, kGateRows) ||
        encode_map(&cached.w_down, w_down, (uint64_t)d.E * d.H, d.I, kGateRows))
      return false;
    if (d.Is > 0 &&
        (encode_map(&cached.w_gu_s, se.gate_up, 2 * (uint64_t)d.Is, d.H, kGateRows) ||
         encode_map(&cached.w_down_s, se.down, (uint64_t)d.H, d.Is, kGateRows)))
      return false;
    last_w = kw;
    have_w = true;
  }
  if (!(have_t && kt == last_t)) {
    have_t = false;
    // token boxes up to the chunk: an item's box covers at most chunk rows;
    // each CTA of a pair loads half of an item's rows, so its boxes are half
    // as high (8 (b + 1) rows for 16 (b + 1) tokens)
    for (int b = 0; b < kTokBoxSizes && kTokBox * (b + 1) <= d.tok_chunk; ++b) {
      const uint32_t rows = (uint32_t)((d.pair ? kTokBox / 2 : kTokBox) * (b + 1));
      if (encode_map(&cached.xp[b], w.xp, slots, d.H, rows) ||
          encode_map(&cached.act[b], w.act, slots, d.I, rows))
        return false;
      if (d.Is > 0 && (encode_map(&cached.xt[b], w.xt, (uint64_t)d.B, d.H, rows) ||
                       encode_map(&cached.act_s[b], w.act_s, (uint64_t)d.B, d.Is, rows)))
        return false;
    }
    last_t = kt;
    have_t = true;
  }
  *maps = cached;
  return true;
}

int decode_impl(const void *hidden, const float *router_w, const int32_t *retained,
                int32_t n_retained, const void *w_gate_up, const void *w_down,
                int32_t top_k, void *out, void *stream, const slimwise_moe_shape *shape,
                void *workspace, size_t workspace_bytes, const slimwise_decode_opts *opts,
                const SharedExpert *shared = nullptr) {
  const int32_t m_ret = retained ? n_retained : (shape ? shape->num_experts : 0);
  int rc = check_shape(shape, top_k, m_ret);
  if (rc) return rc;
  const SharedExpert se = shared ? *shared : SharedExpert{nullptr, nullptr, nullptr, 0};
  if (shared && (se.inter < 64 || se.inter % 64 != 0 || se.inter > 65536))
    return SLIMWISE_ERR_UNSUPPORTED_SHAPE;
  if (shape->num_tokens == 0) return SLIMWISE_OK;
  if (shared) {
    if (!se.gate || !se.gate_up || !se.down) return SLIMWISE_ERR_INVALID_ARG;
    if (!aligned(se.gate, 16) || !aligned(se.gate_up, 16) || !aligned(se.down, 16))
      return SLIMWISE_ERR_UNSUPPORTED_SHAPE;
  }
  if (!hidden || !router_w || !w_gate_up || !w_down || !out) return SLIMWISE_ERR_INVALID_ARG;
  if (!aligned(hidden, 16) || !aligned(router_w, 16) || !aligned(w_gate_up, 16) ||
      !aligned(w_down, 16) || !aligned(out, 16) || (retained && !aligned(retained, 4)))
    return SLIMWISE_ERR_UNSUPPORTED_SHAPE;
  WsLayout L;
  rc = check_workspace(shape, top_k, workspace, workspace_bytes, &L, se.inter);
  if (rc) return rc;
  DeviceInfo di;
  rc = device_info(&di);
  if (rc) return rc;

  Dims d = make_dims(shape, top_k, m_ret, se.inter);
  if (opts) apply_item_form(&d, opts->ffn_items);
  const Ws w = make_ws(workspace, L);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const bool pdl = !(opts && opts->disable_pdl);
  int grid = di.sms;
  if (opts && opts->grid_ctas > 0) grid = opts->grid_ctas;

  FfnMaps maps;
  const uint64_t slots = (uint64_t)d.B * d.k;
  if (!ffn_maps_for(&maps, w_gate_up, w_down, w, d, slots, se)) return SLIMWISE_ERR_CUDA;

  if (launch_route_topk(static_cast<const __nv_bfloat16 *>(hidden), router_w, retained,
                        d, w, pdl, st) != cudaSuccess)
    return SLIMWISE_ERR_CUDA;
  if (launch_group_gather(static_cast<const __nv_bfloat16 *>(hidden), se.gate, d, w, pdl, true,
                          st) != cudaSuccess)
    return SLIMWISE_ERR_CUDA;
  const bool timed = opts && opts->ffn_begin && opts->ffn_end;
  if (timed && cudaEventRecord(static_cast<cudaEvent_t>(opts->ffn_begin), st) != cudaSuccess)
    return SLIMWISE_ERR_CUDA;
  const uint64_t wait_limit = (opts && opts->wait_limit_ns > 0)
                                  ? (uint64_t)opts->wait_limit_ns
                                  : kDefaultWaitLimitNs;
  const int starve = (opts && opts->test_starve_first_down) ? 1 : 0;
  if (launch_expert_ffn(maps, d, w, static_cast<__nv_bfloat16 *>(out), retained, grid,
                        pdl && !timed, st, wait_limit, starve) != cudaSuccess)
    return SLIMWISE_ERR_CUDA;
  // the combine belongs to the timed span: the events bracket the expert FFN
  // and the combine of its outputs
  if (launch_combine(d, w, static_cast<__nv_bfloat16 *>(out), pdl, st) != cudaSuccess)
    return SLIMWISE_ERR_CUDA;
  if (timed && cudaEventRecord(static_cast<cudaEvent_t>(opts->ffn_end), st) != cudaSuccess)
    return SLIMWISE_ERR_CUDA;
  return SLIMWISE_OK;
}

}  // namespace

extern "C" {

const char *slimwise_status_string(int status) {
  switch (status) {
    case SLIMWISE_OK: return "ok";
    case SLIMWISE_ERR_INVALID_ARG: return "invalid argument";
    case SLIMWISE_ERR_UNSUPPORTED_SHAPE: return "unsupported shape or alignment";
    case SLIMWISE_ERR_WORKSPACE: return "workspace too small";
    case SLIMWISE_ERR_CUDA: return "CUDA error";
    case SLIMWISE_ERR_DEVICE: return "device-side error";
    default: return "unknown status";
  }
}

int slimwise_moe_workspace_size(const slimwise_moe_shape *shape, int32_t top_k,
                                size_t *bytes) {
  if (!bytes) return SLIMWISE_ERR_INVALID_ARG;
  int rc = check_shape(shape, top_k, shape ? shape->num_experts : 0);
  if (rc) return rc;
  *bytes = make_layout(shape->num_tokens, shape->hidden, shape->num_experts,
                       shape->inter, top_k)
               .total;
  return SLIMWISE_OK;
}

int slimwise_moe_shared_workspace_size(const slimwise_moe_shape *shape, int32_t top_k,
                                       int32_t inter_shared, size_t *bytes) {
  if (!bytes) return SLIMWISE_ERR_INVALID_ARG;
  int rc = check_shape(shape, top_k, shape ? shape->num_experts : 0);
  if (rc) return rc;
  if (inter_shared < 64 || inter_shared % 64 != 0 || inter_shared > 65536)
    return SLIMWISE_ERR_UNSUPPORTED_SHAPE;
  *bytes = make_layout(shape->num_tokens, shape->hidden, shape->num_experts,
                       shape->inter, top_k, inter_shared)
               .total;
  return SLIMWISE_OK;
}

int slimwise_moe_decode_shared(const void *hidden, const float *router_w,
                               const int32_t *retained_idx, int32_t n_retained,
                               const void *w_gate_up, const void *w_down, int32_t top_k,
                               const float *w_shared_gate, const void *w_shared_gate_up,
                               const void *w_shared_down, int32_t inter_shared, void *out,
                               void *stream, const slimwise_moe_shape *shape,
                               void *workspace, size_t workspace_bytes) {
  const SharedExpert se = {w_shared_gate, w_shared_gate_up, w_shared_down, inter_shared};
  return decode_impl(hidden, router_w, retained_idx, n_retained, w_gate_up, w_down, top_k,
                     out, stream, shape, workspace, workspace_bytes, nullptr, &se);
}

int slimwise_moe_decode_shared_ex(const void *hidden, const float *router_w,
                                  const int32_t *retained_idx, int32_t n_retained,
                                  const void *w_gate_up, const void *w_down, int32_t top_k,
                                  const float *w_shared_gate, const void *w_shared_gate_up,
                                  const void *w_shared_down, int32_t inter_shared, void *out,
                                  void *stream, const slimwise_moe_shape *shape,
                                  void *workspace, size_t workspace_bytes,
                                  const slimwise_decode_opts *opts) {
  const SharedExpert se = {w_shared_gate, w_shared_gate_up, w_shared_down, inter_shared};
  return decode_impl(hidden, router_w, retained_idx, n_retained, w_gate_up, w_down, top_k,
                     out, stream, shape, workspace, workspace_bytes, opts, &se);
}

int slimwise_moe_expert_stats(const void *hidden, const float *router_w,
                              const void *w_gate_up, const void *w_down, int32_t top_k,
                              double *stats, void *out, void *stream,
                              const slimwise_moe_shape *shape, void *workspace,
                              size_t workspace_bytes) {
  int rc = check_shape(shape, top_k, shape ? shape->num_experts : 0);
  if (rc) return rc;
  if (shape->num_tokens == 0) return SLIMWISE_OK;
  if (!stats) return SLIMWISE_ERR_INVALID_ARG;
  if (!aligned(stats, 8)) return SLIMWISE_ERR_UNSUPPORTED_SHAPE;
  // the full-pool layer (its output is the calibration pass's layer output)
  rc = decode_impl(hidden, router_w, nullptr, 0, w_gate_up, w_down, top_k, out, stream, shape,
                   workspace, workspace_bytes, nullptr);
  if (rc) return rc;
  WsLayout L;
  rc = check_workspace(shape, top_k, workspace, workspace_bytes, &L);
  if (rc) return rc;
  const Dims d = make_dims(shape, top_k, shape->num_experts);
  return launch_expert_stats(d, make_ws(workspace, L), stats,
                             reinterpret_cast<cudaStream_t>(stream)) == cudaSuccess
             ? SLIMWISE_OK
             : SLIMWISE_ERR_CUDA;
}

int slimwise_moe_select_retained(const double *stats, int32_t num_experts, int32_t n_retained,
                                 int32_t criterion, int32_t *retained_idx, void *stream) {
  if (num_experts < 1 || num_experts > kMaxExperts) return SLIMWISE_ERR_UNSUPPORTED_SHAPE;
  if (n_retained < 0 || n_retained > num_experts) return SLIMWISE_ERR_INVALID_ARG;
  if (criterion < SLIMWISE_CRITERION_MASS || criterion > SLIMWISE_CRITERION_REAP)
    return SLIMWISE_ERR_INVALID_ARG;
  if (n_retained == 0) return SLIMWISE_OK;
  if (!stats || !retained_idx) return SLIMWISE_ERR_INVALID_ARG;
  if (!aligned(stats, 8) || !aligned(retained_idx, 4)) return SLIMWISE_ERR_UNSUPPORTED_SHAPE;
  return launch_select_retained(stats, num_experts, n_retained, criterion, retained_idx,
                                reinterpret_cast<cudaStream_t>(stream)) == cudaSuccess
             ? SLIMWISE_OK
             : SLIMWISE_ERR_CUDA;
}

int slimwise_moe_compact_layer(const void *w_gate_up, const void *w_down,
                               const float *router_w, const int32_t *retained_idx,
                               int32_t n_retained, const slimwise_moe_shape *shape,
                               void *w_gate_up_c, void *w_down_c, float *router_w_c,
                               int32_t *ids_c, void *stream) {
  if (!shape) return SLIMWISE_ERR_INVALID_ARG;
  // the shape checks of a layer (num_tokens unused; top-1 is always valid)
  slimwise_moe_shape s = *shape;
  s.num_tokens = 0;
  int rc = check_shape(&s, 1, n_retained);
  if (rc) return rc;
  if (!w_gate_up || !w_down || !router_w || !retained_idx || !w_gate_up_c || !w_down_c ||
      !router_w_c || !ids_c)
    return SLIMWISE_ERR_INVALID_ARG;
  if (!aligned(w_gate_up, 16) || !aligned(w_down, 16) || !aligned(router_w, 16) ||
      !aligned(w_gate_up_c, 16) || !aligned(w_down_c, 16) || !aligned(router_w_c, 16) ||
      !aligned(retained_idx, 4) || !aligned(ids_c, 4))
    return SLIMWISE_ERR_UNSUPPORTED_SHAPE;
  DeviceInfo di;
  rc = device_info(&di);
  if (rc) return rc;
  return launch_compact_layer(w_gate_up, w_down, router_w, retained_idx, n_retained,
                              shape->num_experts, shape->hidden, shape->inter, di.sms,
                              w_gate_up_c, w_down_c, router_w_c, ids_c,
                              reinterpret_cast<cudaStream_t>(stream)) == cudaSuccess
             ? SLIMWISE_OK
             : SLIMWISE_ERR_CUDA;
}

int slimwise_moe_decode(const void *hidden, const float *router_w,
                        const int32_t *retained_idx, int32_t n_retained,
                        const void *w_gate_up, const void *w_down, int32_t top_k,
                        void *out, void *stream, const slimwise_moe_shape *shape,
                        void *workspace, size_t workspace_bytes) {
  if (!retained_idx) return SLIMWISE_ERR_INVALID_ARG;
  return decode_impl(hidden, router_w, retained_idx, n_retained, w_gate_up, w_down,
                     top_k, out, stream, shape, workspace, workspace_bytes, nullptr);
}

int slimwise_moe_decode_full(const void *hidden, const float *router_w,
                             const void *w_gate_up, const void *w_down, int32_t top_k,
                             void *out, void *stream, const slimwise_moe_shape *shape,
                             void *workspace, size_t workspace_bytes) {
  return decode_impl(hidden, router_w, nullptr, 0, w_gate_up, w_down, top_k, out, stream,
                     shape, workspace, workspace_bytes, nullptr);
}

int slimwise_moe_decode_ex(const void *hidden, const float *router_w,
                           const int32_t *retained_idx, int32_t n_retained,
                           const void *w_gate_up, const void *w_down, int32_t top_k,
                           void *out, void *stream, const slimwise_moe_shape *shape,
                           void *workspace, size_t workspace_bytes,
                           const slimwise_decode_opts *opts) {
  return decode_impl(hidden, router_w, retained_idx, n_retained, w_gate_up, w_down, top_k,
                     out, stream, shape, workspace, workspace_bytes, opts);
}

int slimwise_moe_route(const void *hidden, const float *router_w,
                       const int32_t *retained_idx, int32_t n_retained, int32_t top_k,
                       void *stream, const slimwise_moe_shape *shape, void *workspace,
                       size_t workspace_bytes, int32_t *topk_idx, float *topk_gate,
                       int32_t *counts, int32_t *offsets, int32_t *union_ids,
                       int32_t *union_size, int32_t *perm, int32_t *pos) {
  const int32_t m_ret = retained_idx ? n_retained : (shape ? shape->num_experts : 0);
  int rc = check_shape(shape, top_k, m_ret);
  if (rc) return rc;
  if (shape->num_tokens == 0) return SLIMWISE_OK;
  if (!hidden || !router_w) return SLIMWISE_ERR_INVALID_ARG;
  if (!aligned(hidden, 16) || !aligned(router_w, 16)) return SLIMWISE_ERR_UNSUPPORTED_SHAPE;
  WsLayout L;
  rc = check_workspace(shape, top_k, workspace, workspace_bytes, &L);
  if (rc) return rc;
  DeviceInfo di;
  rc = device_info(&di);
  if (rc) return rc;
  const Dims d = make_dims(shape, top_k, m_ret);
  const Ws w = make_ws(workspace, L);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (launch_route_topk(static_cast<const __nv_bfloat16 *>(hidden), router_w, retained_idx,
                        d, w, false, st) != cudaSuccess ||
      launch_group_gather(static_cast<const __nv_bfloat16 *>(hidden), nullptr, d, w, false, false,
                          st) != cudaSuccess)
    return SLIMWISE_ERR_CUDA;
  const size_t slots = (size_t)d.B * d.k;
  rc = copy_out(topk_idx, w.topk_idx, slots * 4, st);
  if (!rc) rc = copy_out(topk_gate, w.topk_gate, slots * 4, st);
  if (!rc) rc = copy_group_outputs(w, d, st, counts, offsets, union_ids, union_size, perm, pos);
  return rc;
}

int slimwise_moe_group(const int32_t *topk_idx, int32_t top_k, void *stream,
                       const slimwise_moe_shape *shape, void *workspace,
                       size_t workspace_bytes, int32_t *counts, int32_t *offsets,
                       int32_t *union_ids, int32_t *union_size, int32_t *perm,
                       int32_t *pos) {
  int rc = check_shape(shape, top_k, shape ? shape->num_experts : 0);
  if (rc) return rc;
  if (shape->num_tokens == 0) return SLIMWISE_OK;
  if (!topk_idx) return SLIMWISE_ERR_INVALID_ARG;
  WsLayout L;
  rc = check_workspace(shape, top_k, workspace, workspace_bytes, &L);
  if (rc) return rc;
  DeviceInfo di;
  rc = device_info(&di);
  if (rc) return rc;
  const Dims d = make_dims(shape, top_k, shape->num_experts);
  const Ws w = make_ws(workspace, L);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const size_t slots = (size_t)d.B * d.k;
  if (cudaMemsetAsync(w.ctrl + kCtrlErr, 0, 4, st) != cudaSuccess ||
      cudaMemcpyAsync(w.topk_idx, topk_idx, slots * 4, cudaMemcpyDeviceToDevice, st) !=
          cudaSuccess ||
      launch_group_gather(nullptr, nullptr, d, w, false, false, st) != cudaSuccess)
    return SLIMWISE_ERR_CUDA;
  return copy_group_outputs(w, d, st, counts, offsets, union_ids, union_size, perm, pos);
}

int slimwise_moe_device_status(const void *workspace, void *stream, int32_t *flags) {
  if (!workspace || !flags) return SLIMWISE_ERR_INVALID_ARG;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  int32_t v = 0;
  const int32_t *src = static_cast<const int32_t *>(workspace) + kCtrlErr;  // ctrl is first
  if (cudaMemcpyAsync(&v, src, 4, cudaMemcpyDeviceToHost, st) != cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess)
    return SLIMWISE_ERR_CUDA;
  *flags = v;
  return v ? SLIMWISE_ERR_DEVICE : SLIMWISE_OK;
}

}  // extern "C"
