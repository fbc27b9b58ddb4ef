// compact_layer.cu -- the compact (pruned) checkpoint of one MoE layer.
//
// A decode instance that serves from the pruned pool K' needs only the m'
// retained experts' weights and router rows (SlimWise Sec. 3.1: the Eq. 2
// router mask and a checkpoint holding only K' are two forms of the same
// layer).  These kernels build that form on the device from the full layer:
//   compact_ids_kernel   the retained ids in ascending order (one CTA; the
//                        rank of an id is the number of smaller ids), so
//                        top-k ties in the compact numbering still go to the
//                        lowest original id;
//   compact_copy_kernel  for compact expert j = original expert ids[j]: its
//                        [2I, H] gate/up rows, [H, I] down rows and router
//                        row, 16 bytes per thread per step, with streaming
//                        (evict-first) loads and stores -- a pure copy, bound
//                        by HBM at 2 x (m' x expert bytes).
// A repeated or out-of-range id sets every entry of ids to -1, and then the
// copy kernel writes nothing.
#include "common.cuh"

namespace slimwise {

constexpr int kIdsThreads = 1024;   // >= kMaxExperts: one id per thread
constexpr int kCopyThreads = 256;
constexpr int kCopyUnroll = 4;      // 16-byte loads in flight per thread

__global__ void __launch_bounds__(kIdsThreads)
    compact_ids_kernel(const int32_t *__restrict__ retained, int m, int E,
                       int32_t *__restrict__ ids_c) {
  __shared__ int ids[kMaxExperts];
  __shared__ int bad;
  const int i = threadIdx.x;
  if (i == 0) bad = 0;
  if (i < m) ids[i] = retained[i];
  __syncthreads();
  int rank = 0, same = 0;
  if (i < m) {
    const int e = ids[i];
    for (int j = 0; j < m; ++j) {
      rank += ids[j] < e ? 1 : 0;
      same += ids[j] == e ? 1 : 0;
    }
    if (e < 0 || e >= E || same != 1) bad = 1;
  }
  __syncthreads();
  if (i < m) {
    if (bad) ids_c[i] = -1;
    else ids_c[rank] = ids[i];
  }
}

// Copy of `n` 16-byte vectors from src to dst, grid-strided over the CTAs of
// one compact expert; kCopyUnroll loads are issued before their stores.
__device__ __forceinline__ void copy_vecs(const uint4 *__restrict__ src, uint4 *__restrict__ dst,
                                          size_t n, size_t t0, size_t stride) {
  size_t i = t0;
  for (; i + (kCopyUnroll - 1) * stride < n; i += kCopyUnroll * stride) {
    uint4 v[kCopyUnroll];
#pragma unroll
    for (int u = 0; u < kCopyUnroll; ++u) v[u] = __ldcs(src + i + u * stride);
#pragma unroll
    for (int u = 0; u < kCopyUnroll; ++u) __stcs(dst + i + u * stride, v[u]);
  }
  for (; i < n; i += stride) __stcs(dst + i, __ldcs(src + i));
}

// blockIdx.y = compact expert j; the gridDim.x CTAs of row j split its bytes.
__global__ void __launch_bounds__(kCopyThreads)
    compact_copy_kernel(const uint4 *__restrict__ w_gu, const uint4 *__restrict__ w_d,
                        const uint4 *__restrict__ wr, const int32_t *__restrict__ ids_c,
                        size_t gu_vecs, size_t d_vecs, size_t wr_vecs, uint4 *__restrict__ gu_c,
                        uint4 *__restrict__ d_c, uint4 *__restrict__ wr_c) {
  const size_t j = blockIdx.y;
  const int e = ids_c[j];
  if (e < 0) return;  // repeated or out-of-range ids: nothing is copied
  const size_t t0 = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  const size_t stride = (size_t)gridDim.x * blockDim.x;
  copy_vecs(w_gu + (size_t)e * gu_vecs, gu_c + j * gu_vecs, gu_vecs, t0, stride);
  copy_vecs(w_d + (size_t)e * d_vecs, d_c + j * d_vecs, d_vecs, t0, stride);
  copy_vecs(wr + (size_t)e * wr_vecs, wr_c + j * wr_vecs, wr_vecs, t0, stride);
}

cudaError_t launch_compact_layer(const void *w_gate_up, const void *w_down, const float *router_w,
                                 const int32_t *retained, int m, int E, int H, int I, int sms,
                                 void *w_gate_up_c, void *w_down_c, float *router_w_c,
                                 int32_t *ids_c, cudaStream_t stream) {
  compact_ids_kernel<<<1, kIdsThreads, 0, stream>>>(retained, m, E, ids_c);
  cudaError_t err = cudaGetLastError();
  if (err != cudaSuccess) return err;
  // bytes per expert: 2I x H and H x I bf16, H fp32 -- multiples of 16
  // bytes, since H is a multiple of 128 and I of 64
  const size_t gu_vecs = (size_t)2 * I * H * 2 / 16;
  const size_t d_vecs = (size_t)H * I * 2 / 16;
  const size_t wr_vecs = (size_t)H * 4 / 16;
  // about four CTAs per SM over the whole copy, at least one per expert
  int per_expert = (4 * sms + m - 1) / m;
  if (per_expert < 1) per_expert = 1;
  const dim3 grid((unsigned)per_expert, (unsigned)m);
  compact_copy_kernel<<<grid, kCopyThreads, 0, stream>>>(
      static_cast<const uint4 *>(w_gate_up), static_cast<const uint4 *>(w_down),
      reinterpret_cast<const uint4 *>(router_w), ids_c, gu_vecs, d_vecs, wr_vecs,
      static_cast<uint4 *>(w_gate_up_c), static_cast<uint4 *>(w_down_c),
      reinterpret_cast<uint4 *>(router_w_c));
  return cudaGetLastError();
}

}  // namespace slimwise
