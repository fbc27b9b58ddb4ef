// group_gather.cu -- grouping of the B*k routed (token, slot) pairs by expert
// and gather of the hidden rows into that grouped order.
//
// A decode step must read the weights of the union of experts selected
// across the batch (SlimWise Sec. 2.1, Eq. 1).  This kernel turns the top-k
// selections into:
//   counts[e]  histogram of selections,
//   offsets    exclusive scan of counts (expert ascending),
//   union_ids  selected experts ascending, union size U,
//   perm/pos   grouped order of the slots: (expert asc, token asc),
//   entries    the FFN kernel's work list: one entry per (expert, chunk of
//              at most tok_chunk tokens),
//   xp         hidden rows copied into grouped order, so the FFN kernel can
//              stream each expert's tokens with plain 2-D TMA boxes.
// With a shared expert (Sec. 3.3) it also computes each token's sigmoid gate
// s_t = 1 / (1 + exp(-w_sg . x_t)), the dot product in the canonical order of
// the router logits, and lists the shared expert's work entries (the batch in
// token order, in chunks) ahead of the routed ones.
// Every CTA recomputes the histogram of the whole batch (B*k ids, a few KB
// from L2) so the rank of a slot inside its expert, its token-order prefix
// count, is known without a grid-wide barrier; integer counts make the
// result independent of atomic arrival order.
#include "common.cuh"

namespace slimwise {

// Tokens per CTA: one up to 64 tokens, two above.  Fewer tokens per CTA
// spread the grouped-row copy over more SMs (one against two: up to 1.1 us a
// step faster at B = 8-64), but every CTA recounts the whole batch's
// selections, and above 64 tokens the extra CTAs cost more (B = 256: 0.9 us,
// B = 512: 2 us slower); four per CTA was slower at every size.
inline int group_tokens_per_cta(int B) { return B <= 64 ? 1 : 2; }
constexpr int kGroupThreads = 512;

// Exclusive scan of vals[0..n) (n <= kMaxExperts) into outp[0..n], by one
// warp; returns the total.  Each lane scans a contiguous run.
__device__ int warp_exclusive_scan(const int *vals, int *outp, int n, int lane) {
  const int per = (n + 31) / 32;
  const int lo = min(n, lane * per), hi = min(n, lo + per);
  int local = 0;
  for (int i = lo; i < hi; ++i) local += vals[i];
  int incl = local;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    int o = __shfl_up_sync(0xFFFFFFFFu, incl, off);
    if (lane >= off) incl += o;
  }
  int run = incl - local;
  for (int i = lo; i < hi; ++i) {
    outp[i] = run;
    run += vals[i];
  }
  const int total = __shfl_sync(0xFFFFFFFFu, incl, 31);
  if (lane == 0) outp[n] = total;
  return total;
}

template <int kGroupTokens>
__global__ void __launch_bounds__(kGroupThreads)
    group_gather_kernel(const __nv_bfloat16 *__restrict__ hidden,
                        const float *__restrict__ w_sg, Dims d, Ws ws, int do_gather) {
  __shared__ int cnt_all[kMaxExperts];
  __shared__ int cnt_before[kMaxExperts];
  __shared__ int union_flag[kMaxExperts];
  __shared__ int offs[kMaxExperts + 1];
  __shared__ int flag_scan[kMaxExperts + 1];
  __shared__ int chunk_cnt[kMaxExperts];
  __shared__ int entry_base[kMaxExperts + 1];
  __shared__ int my_pos[kGroupTokens * kMaxTopK];
  __shared__ int my_ids[kGroupTokens * kMaxTopK];
  __shared__ int bad;

  // Wait for the routing kernel's results; then let the FFN kernel's CTAs
  // start their prologue.
  pdl_wait_primary();
  pdl_launch_dependents();
#ifdef SLIMWISE_TRACE
  const int tr_step = ws.ctrl[kCtrlTraceStep] - 1;
  if (blockIdx.x == 0 && threadIdx.x == 0) trace_stamp(ws, tr_step, kTrGroupStart);
#endif

  const int B = d.B, k = d.k, E = d.E, H = d.H;
  const int S = B * k;
  const int t0 = blockIdx.x * kGroupTokens;
  const int t1 = min(B, t0 + kGroupTokens);
  const int nt = t1 - t0;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int vecs = H / 8;  // 16-byte vectors per hidden row

  // This CTA's hidden rows go into registers first, so that their loads
  // overlap the histogram below (up to kPre vectors per thread).
  constexpr int kPre = 4;
  const bool early = do_gather && nt * vecs <= kPre * (int)blockDim.x;
  uint4 hv[kPre];
  if (early) {
#pragma unroll
    for (int u = 0; u < kPre; ++u) {
      const int i = tid + u * blockDim.x;
      if (i < nt * vecs)
        hv[u] = __ldg(reinterpret_cast<const uint4 *>(hidden + (size_t)(t0 + i / vecs) * H) + i % vecs);
    }
  }

  for (int e = tid; e < E; e += blockDim.x) {
    cnt_all[e] = 0;
    cnt_before[e] = 0;
  }
  if (tid == 0) bad = 0;
  __syncthreads();
  const int nslots = nt * k;
  // each thread's selections are loaded together, then counted
  constexpr int kHistBatch = 8;
  for (int s0 = tid; s0 < S; s0 += kHistBatch * blockDim.x) {
    int ev[kHistBatch];
#pragma unroll
    for (int u = 0; u < kHistBatch; ++u) {
      const int s = s0 + u * blockDim.x;
      ev[u] = s < S ? ws.topk_idx[s] : 0;
    }
#pragma unroll
    for (int u = 0; u < kHistBatch; ++u) {
      const int s = s0 + u * blockDim.x;
      if (s < S) {
        int e = ev[u];
        if (e < 0 || e >= E) {  // only possible for caller-given selections
          bad = SLIMWISE_DEVERR_BAD_TOPK;
          e = min(max(e, 0), E - 1);
        }
        atomicAdd(&cnt_all[e], 1);
        if (s < t0 * k) atomicAdd(&cnt_before[e], 1);
        else if (s < t1 * k) my_ids[s - t0 * k] = e;
      }
    }
  }
  __syncthreads();
  // offsets of the experts; union flags and work-entry counts (every CTA has
  // the whole histogram, so each can publish its share of the results)
  for (int e = tid; e < E; e += blockDim.x) {
    union_flag[e] = cnt_all[e] > 0 ? 1 : 0;
    chunk_cnt[e] = (cnt_all[e] + d.tok_chunk - 1) / d.tok_chunk;
  }
  __syncthreads();
  if (warp == 0) warp_exclusive_scan(cnt_all, offs, E, lane);
  if (warp == 1) warp_exclusive_scan(union_flag, flag_scan, E, lane);
  if (warp == 2) warp_exclusive_scan(chunk_cnt, entry_base, E, lane);
  __syncthreads();

  // Grouped position of each of this CTA's slots: offset of the expert plus
  // the number of earlier tokens that selected it (tokens before this CTA's
  // range, then earlier tokens of the range).
  for (int i = tid; i < nslots; i += blockDim.x) {
    const int e = my_ids[i];
    int rank = cnt_before[e];
    for (int s = 0; s < (i / k) * k; ++s) rank += (my_ids[s] == e) ? 1 : 0;
    my_pos[i] = offs[e] + rank;
  }
  __syncthreads();
  for (int i = tid; i < nslots; i += blockDim.x) {
    const int s = t0 * k + i, p = my_pos[i];
    ws.pos[s] = p;
    ws.perm[p] = s;
  }
  if (early) {
    // each token row, already in registers, goes to its k grouped positions
#pragma unroll
    for (int u = 0; u < kPre; ++u) {
      const int i = tid + u * blockDim.x;
      if (i < nt * vecs) {
        const int tt = i / vecs, vv = i % vecs;
        for (int j = 0; j < k; ++j)
          reinterpret_cast<uint4 *>(ws.xp + (size_t)my_pos[tt * k + j] * H)[vv] = hv[u];
        // token-order copy for the shared expert (a stable address to map)
        if (d.Is > 0) reinterpret_cast<uint4 *>(ws.xt + (size_t)(t0 + tt) * H)[vv] = hv[u];
      }
    }
  } else if (do_gather) {
    // wide rows: loaded here, four vectors per thread in flight
    constexpr int kVec = 4;
    for (int i0 = tid; i0 < nt * vecs; i0 += kVec * blockDim.x) {
      uint4 v[kVec];
      int tt[kVec], vv[kVec];
#pragma unroll
      for (int u = 0; u < kVec; ++u) {
        const int i = i0 + u * blockDim.x;
        tt[u] = i / vecs;
        vv[u] = i - tt[u] * vecs;
        if (i < nt * vecs)
          v[u] = __ldg(reinterpret_cast<const uint4 *>(hidden + (size_t)(t0 + tt[u]) * H) + vv[u]);
      }
#pragma unroll
      for (int u = 0; u < kVec; ++u) {
        if (i0 + u * blockDim.x < nt * vecs) {
          for (int j = 0; j < k; ++j)
            reinterpret_cast<uint4 *>(ws.xp + (size_t)my_pos[tt[u] * k + j] * H)[vv[u]] = v[u];
          if (d.Is > 0) reinterpret_cast<uint4 *>(ws.xt + (size_t)(t0 + tt[u]) * H)[vv[u]] = v[u];
        }
      }
    }
  }
  // shared-expert gate of this CTA's tokens: warp w takes token t0 + w; lane
  // l accumulates elements 128c + 4l + q (c, q ascending) with fused
  // multiply-adds, then an xor butterfly over the lanes
  if (d.Is > 0 && warp < nt) {
    const __nv_bfloat16 *xr = hidden + (size_t)(t0 + warp) * H;
    float p = 0.0f;
    for (int c = 0; c < H / 128; ++c) {
      const int h = 128 * c + 4 * lane;
      const uint2 xv = *reinterpret_cast<const uint2 *>(xr + h);
      const float4 wv = *reinterpret_cast<const float4 *>(w_sg + h);
      p = fmaf(__uint_as_float(xv.x << 16), wv.x, p);
      p = fmaf(__uint_as_float(xv.x & 0xFFFF0000u), wv.y, p);
      p = fmaf(__uint_as_float(xv.y << 16), wv.z, p);
      p = fmaf(__uint_as_float(xv.y & 0xFFFF0000u), wv.w, p);
    }
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) p = p + __shfl_xor_sync(0xFFFFFFFFu, p, off);
    if (lane == 0) ws.shared_gate[t0 + warp] = 1.0f / (1.0f + expf(-p));
  }

  // The batch-wide results and the FFN work list, each expert written by one
  // thread of the grid.  Entries [0, n_se) are the shared expert's (expert
  // -1, token order); the routed ones follow.
  const int U = flag_scan[E];
  const int n_entries = entry_base[E];
  const int n_se = d.S;
  const int gtid = blockIdx.x * blockDim.x + tid, gstride = gridDim.x * blockDim.x;
  for (int e = gtid; e < E; e += gstride) {
    ws.counts[e] = cnt_all[e];
    ws.offsets[e] = offs[e];
    if (union_flag[e]) ws.union_ids[flag_scan[e]] = e;
    if (e >= U) ws.union_ids[e] = -1;
    const int n_e = offs[e + 1] - offs[e];
    for (int c = 0; c < chunk_cnt[e]; ++c) {
      const int base = c * d.tok_chunk;
      ws.entries[n_se + entry_base[e] + c] =
          make_int4(e, offs[e] + base, min(d.tok_chunk, n_e - base), 0);
    }
  }
  for (int sidx = gtid; sidx < n_se; sidx += gstride)
    ws.entries[sidx] = make_int4(-1, sidx * d.tok_chunk, min(d.tok_chunk, B - sidx * d.tok_chunk), 0);
  for (int i = gtid; i < n_se + n_entries; i += gstride) ws.entry_done[i] = 0;
  if (blockIdx.x == 0 && tid == 0) {
    const int t1_items = gate_up_tiles(d);
    const int t2_items = down_tiles(d);
    const int t1s_items = d.Is / kGateRows;
    ws.offsets[E] = offs[E];
    ws.ctrl[kCtrlUnionSize] = U;
    ws.ctrl[kCtrlNumEntries] = n_se + n_entries;
    ws.ctrl[kCtrlItems1] = n_entries * t1_items;
    ws.ctrl[kCtrlTotalItems] = n_se * (t1s_items + t2_items) + n_entries * (t1_items + t2_items);
    ws.ctrl[kCtrlWorkCounter] = 0;
  }
  __syncthreads();
  if (blockIdx.x == 0 && tid == 0 && bad) atomicOr(&ws.ctrl[kCtrlErr], bad);
#ifdef SLIMWISE_TRACE
  if (blockIdx.x == 0 && tid == 0) trace_stamp(ws, tr_step, kTrGroupEnd);
#endif
}

cudaError_t launch_group_gather(const __nv_bfloat16 *hidden, const float *w_shared_gate,
                                Dims d, Ws ws, bool pdl, bool gather, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  const int tpc = group_tokens_per_cta(d.B);
  cfg.gridDim = dim3((d.B + tpc - 1) / tpc);
  cfg.blockDim = dim3(kGroupThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  if (tpc == 1)
    return cudaLaunchKernelEx(&cfg, group_gather_kernel<1>, hidden, w_shared_gate, d, ws,
                              gather ? 1 : 0);
  return cudaLaunchKernelEx(&cfg, group_gather_kernel<2>, hidden, w_shared_gate, d, ws,
                            gather ? 1 : 0);
}

}  // namespace slimwise
