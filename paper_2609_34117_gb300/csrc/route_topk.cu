// route_topk.cu -- router logits over the retained pool, top-k and
// renormalised gates (SlimWise Sec. 3.1, Eq. 2 and the renormalisation that
// follows it).
//
// One CTA handles kRouteTokens tokens against every retained expert.  Logits
// follow the canonical fp32 order: lane l of a warp owns elements
// 128c + 4l + q (q = 0..3) of every 128-wide chunk c, accumulated with fused
// multiply-adds in (c, q) order, then the 32 lane partials are combined by an
// xor butterfly (offsets 16, 8, 4, 2, 1).  The pruned experts are never
// evaluated: restricting top-k to K' is the Eq. 2 mask with tau = -inf, with
// no separate masking pass.  Top-k is a warp-wide arg-max repeated k times
// on a 64-bit key (order-preserving logit bits, then the complemented expert
// id), so ties go to the lowest original id whatever the order of K'.
#include "common.cuh"

namespace slimwise {

constexpr int kRouteTokens = 4;
constexpr int kRouteThreads = 512;
constexpr int kRouteWarps = kRouteThreads / 32;

// Order-preserving map of an fp32 value to uint32 (-0 folded onto +0).
__device__ __forceinline__ uint32_t logit_order_bits(float z) {
  uint32_t b = __float_as_uint(z);
  if ((b << 1) == 0u) b = 0u;
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float logit_from_order_bits(uint32_t o) {
  uint32_t b = (o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o;
  return __uint_as_float(b);
}

__global__ void __launch_bounds__(kRouteThreads)
    route_topk_kernel(const __nv_bfloat16 *__restrict__ hidden,
                      const float *__restrict__ router_w,
                      const int32_t *__restrict__ retained, Dims d, Ws ws) {
  extern __shared__ __align__(16) unsigned char smem[];
  const int H = d.H, m = d.m_ret, k = d.k;
  __nv_bfloat16 *xs = reinterpret_cast<__nv_bfloat16 *>(smem);
  float *zs = reinterpret_cast<float *>(smem + (size_t)kRouteTokens * H * 2);
  int32_t *ids = reinterpret_cast<int32_t *>(zs + (size_t)kRouteTokens * m);

  // Let the grouping kernel become resident; it waits for this grid to end.
  pdl_launch_dependents();

  const int t0 = blockIdx.x * kRouteTokens;
  const int nt = min(kRouteTokens, d.B - t0);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  // Retained ids, clamped into [0, E) so a bad id cannot fault; CTA 0 reports
  // bad and repeated ids and resets the error word of this call.
  for (int r = threadIdx.x; r < m; r += blockDim.x) {
    int e = retained ? retained[r] : r;
    ids[r] = min(max(e, 0), d.E - 1);
  }
  if (blockIdx.x == 0) {
    __shared__ uint32_t seen[kMaxExperts / 32];
    __shared__ int bad;
    for (int i = threadIdx.x; i < kMaxExperts / 32; i += blockDim.x) seen[i] = 0;
    if (threadIdx.x == 0) bad = 0;
    __syncthreads();
    for (int r = threadIdx.x; r < m; r += blockDim.x) {
      int e = retained ? retained[r] : r;
      if (e < 0 || e >= d.E) {
        atomicOr(&bad, SLIMWISE_DEVERR_BAD_RETAINED);
      } else {
        uint32_t bit = 1u << (e & 31);
        if (atomicOr(&seen[e >> 5], bit) & bit)
          atomicOr(&bad, SLIMWISE_DEVERR_DUPLICATE_RETAINED);
      }
    }
    __syncthreads();
    if (threadIdx.x == 0) ws.ctrl[kCtrlErr] = bad;
  }

  // Hidden rows of this CTA's tokens (16-byte vectors).
  const int vecs = H / 8;
  for (int i = threadIdx.x; i < nt * vecs; i += blockDim.x) {
    int t = i / vecs, v = i - t * vecs;
    reinterpret_cast<uint4 *>(xs)[(size_t)t * vecs + v] =
        reinterpret_cast<const uint4 *>(hidden + (size_t)(t0 + t) * H)[v];
  }
  __syncthreads();

  // Logits: warp per retained expert, all tokens of the CTA at once.
  for (int r = warp; r < m; r += kRouteWarps) {
    const float *wrow = router_w + (size_t)ids[r] * H;
    float p[kRouteTokens];
#pragma unroll
    for (int t = 0; t < kRouteTokens; ++t) p[t] = 0.0f;
#pragma unroll 4
    for (int c = 0; c < H / 128; ++c) {
      const float4 w4 = __ldg(reinterpret_cast<const float4 *>(wrow + 128 * c + 4 * lane));
#pragma unroll
      for (int t = 0; t < kRouteTokens; ++t) {
        if (t < nt) {
          const uint2 xr = *reinterpret_cast<const uint2 *>(xs + (size_t)t * H + 128 * c + 4 * lane);
          const float x0 = __uint_as_float(xr.x << 16);
          const float x1 = __uint_as_float(xr.x & 0xFFFF0000u);
          const float x2 = __uint_as_float(xr.y << 16);
          const float x3 = __uint_as_float(xr.y & 0xFFFF0000u);
          p[t] = fmaf(x0, w4.x, p[t]);
          p[t] = fmaf(x1, w4.y, p[t]);
          p[t] = fmaf(x2, w4.z, p[t]);
          p[t] = fmaf(x3, w4.w, p[t]);
        }
      }
    }
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1)
#pragma unroll
      for (int t = 0; t < kRouteTokens; ++t)
        p[t] = p[t] + __shfl_xor_sync(0xFFFFFFFFu, p[t], off);
    if (lane == 0)
#pragma unroll
      for (int t = 0; t < kRouteTokens; ++t)
        if (t < nt) zs[(size_t)t * m + r] = p[t];
  }
  __syncthreads();

  // Top-k and gates: warp per token.
  if (warp < nt) {
    const int t = t0 + warp;
    const float *zt = zs + (size_t)warp * m;
    uint32_t taken = 0;  // bit i: candidate r = lane + 32 i already selected
    float my_z = 0.0f;
    int my_e = 0;
    for (int j = 0; j < k; ++j) {
      unsigned long long best = 0ull;
      int i = 0;
      for (int r = lane; r < m; r += 32, ++i) {
        if ((taken >> i) & 1u) continue;
        unsigned long long key =
            ((unsigned long long)logit_order_bits(zt[r]) << 32) |
            (unsigned long long)(0xFFFFFFFFu - (uint32_t)ids[r]);
        best = key > best ? key : best;
      }
#pragma unroll
      for (int off = 16; off >= 1; off >>= 1) {
        unsigned long long o = __shfl_xor_sync(0xFFFFFFFFu, best, off);
        best = o > best ? o : best;
      }
      // best == 0 only when fewer than k distinct candidates exist (repeated
      // retained ids, already reported); fall back to a valid id.
      const int e_sel = best ? (int)(0xFFFFFFFFu - (uint32_t)(best & 0xFFFFFFFFull)) : ids[0];
      i = 0;
      for (int r = lane; r < m; r += 32, ++i)
        if (ids[r] == e_sel && !((taken >> i) & 1u)) taken |= 1u << i;
      if (lane == j) {
        my_z = logit_from_order_bits((uint32_t)(best >> 32));
        my_e = e_sel;
      }
    }
    // g_j = exp(z_j - z_1) / sum_j' exp(z_j' - z_1), the sum in j order.
    const float z1 = __shfl_sync(0xFFFFFFFFu, my_z, 0);
    const float w = (lane < k) ? expf(my_z - z1) : 0.0f;
    float denom = 0.0f;
    for (int j = 0; j < k; ++j) denom += __shfl_sync(0xFFFFFFFFu, w, j);
    if (lane < k) {
      ws.topk_idx[(size_t)t * k + lane] = my_e;
      ws.topk_gate[(size_t)t * k + lane] = w / denom;
    }
  }
}

size_t route_smem_bytes(const Dims &d) {
  return (size_t)kRouteTokens * d.H * 2 + (size_t)kRouteTokens * d.m_ret * 4 +
         (size_t)d.m_ret * 4;
}

cudaError_t launch_route_topk(const __nv_bfloat16 *hidden, const float *router_w,
                              const int32_t *retained, Dims d, Ws ws,
                              cudaStream_t stream) {
  const size_t smem = route_smem_bytes(d);
  cudaError_t err = cudaFuncSetAttribute(
      route_topk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (err != cudaSuccess) return err;
  const int grid = (d.B + kRouteTokens - 1) / kRouteTokens;
  route_topk_kernel<<<grid, kRouteThreads, smem, stream>>>(hidden, router_w,
                                                           retained, d, ws);
  return cudaGetLastError();
}

}  // namespace slimwise
