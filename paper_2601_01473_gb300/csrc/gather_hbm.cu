// gather_hbm.cu -- block-wise feature gathering from HBM-resident features
// (Algorithm 1's gathering loop, Sec. 3.4 (2)).
//
// The final frontier bucket lists every gathered node once per minibatch, in
// (tile, minibatch, id) order, with its output row.  Tiles never straddle a
// feature block, so walking the bucket in order visits each feature block
// once for all minibatches: a row requested by several minibatches is read
// from HBM once and served from L2 afterwards.  Rows are copied as 16-byte
// vectors (bit-exact, no float conversion); a group of row_bytes/16 lanes
// moves one row, each lane keeping U rows in flight; output stores are
// streaming (evict-first) so they do not push the feature rows out of L2.
#include "common.cuh"
#include "internal.h"

namespace agnes {

namespace {

constexpr int kThreads = 256;
// CTAs per SM of the gather (0: as many as fit) and rows in flight per lane.
// A few CTAs with several rows each keep HBM busy and leave the rest of each
// SM to the kernels of the next hyperbatch, which run beside the gather when
// two hyperbatches are in flight.
constexpr int kGatherCtasPerSm = 3;
constexpr int kU = 8;

// LPR lanes per row, row = LPR 16-byte vectors, U rows in flight per lane.
template <int LPR, int U>
__global__ void __launch_bounds__(kThreads)
gather_vec_kernel(const uint4* __restrict__ feats, const int32_t* __restrict__ fb_id,
                  const int32_t* __restrict__ fb_pos, const int32_t* total_ptr,
                  uint4* __restrict__ out, const int32_t* status) {
  grid_dep_wait();
  if (failed(status)) return;
  constexpr int kRowsPerWarp = 32 / LPR;
  constexpr int kStep = kRowsPerWarp * U;
  const int64_t total = *total_ptr;
  const int lane = lane_id();
  const int sub = lane / LPR, l = lane % LPR;
  const int64_t warp0 = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t r0 = warp0 * kStep; r0 < total; r0 += nwarps * kStep) {
    uint4 v[U];
    int32_t g[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t i = r0 + u * kRowsPerWarp + sub;
      g[u] = -1;
      if (i < total) {
        const int32_t id = __ldg(fb_id + i);
        g[u] = __ldg(fb_pos + i);
        v[u] = __ldg(feats + (int64_t)id * LPR + l);
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u)
      if (g[u] >= 0) __stcs(out + (int64_t)g[u] * LPR + l, v[u]);
  }
}

// Any row size that is a multiple of 16 bytes: one warp per row.
__global__ void __launch_bounds__(kThreads)
gather_rows_kernel(const uint4* __restrict__ feats, int64_t vecs, const int32_t* __restrict__ fb_id,
                   const int32_t* __restrict__ fb_pos, const int32_t* total_ptr,
                   uint4* __restrict__ out, const int32_t* status) {
  grid_dep_wait();
  if (failed(status)) return;
  const int64_t total = *total_ptr;
  const int lane = lane_id();
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t i = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5; i < total; i += nwarps) {
    const int64_t src = (int64_t)__ldg(fb_id + i) * vecs;
    const int64_t dst = (int64_t)__ldg(fb_pos + i) * vecs;
    for (int64_t c = lane; c < vecs; c += 32) __stcs(out + dst + c, __ldg(feats + src + c));
  }
}

// Rows whose size is not a multiple of 16 bytes: byte copy, one warp per row.
__global__ void __launch_bounds__(kThreads)
gather_bytes_kernel(const uint8_t* __restrict__ feats, int64_t row_bytes,
                    const int32_t* __restrict__ fb_id, const int32_t* __restrict__ fb_pos,
                    const int32_t* total_ptr, uint8_t* __restrict__ out, const int32_t* status) {
  grid_dep_wait();
  if (failed(status)) return;
  const int64_t total = *total_ptr;
  const int lane = lane_id();
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t i = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5; i < total; i += nwarps) {
    const int64_t src = (int64_t)__ldg(fb_id + i) * row_bytes;
    const int64_t dst = (int64_t)__ldg(fb_pos + i) * row_bytes;
    for (int64_t c = lane; c < row_bytes; c += 32) out[dst + c] = __ldg(feats + src + c);
  }
}

int gather_grid(const void* kernel, int num_sms) {
  const int g = resident_grid(kernel, kThreads, num_sms);
  return kGatherCtasPerSm > 0 && g > kGatherCtasPerSm * num_sms ? kGatherCtasPerSm * num_sms : g;
}

}  // namespace

cudaError_t launch_gather(const void* feats, int64_t row_bytes, const int32_t* fb_id,
                          const int32_t* fb_pos, const int32_t* total, void* out,
                          const int32_t* status, int num_sms, cudaStream_t st) {
  const bool aligned = (row_bytes % 16 == 0) && ((uintptr_t)feats % 16 == 0) &&
                       ((uintptr_t)out % 16 == 0);
  if (aligned) {
    const int64_t vecs = row_bytes / 16;
    const uint4* f = (const uint4*)feats;
    uint4* o = (uint4*)out;
#define AGNES_GRID(KERNEL) gather_grid((const void*)KERNEL, num_sms), kThreads, 0, st
    if (vecs == 8)
      gather_vec_kernel<8, kU><<<AGNES_GRID((gather_vec_kernel<8, kU>))>>>(f, fb_id, fb_pos, total,
                                                                           o, status);
    else if (vecs == 16)
      gather_vec_kernel<16, kU><<<AGNES_GRID((gather_vec_kernel<16, kU>))>>>(f, fb_id, fb_pos,
                                                                             total, o, status);
    else if (vecs == 32)
      gather_vec_kernel<32, kU><<<AGNES_GRID((gather_vec_kernel<32, kU>))>>>(f, fb_id, fb_pos,
                                                                             total, o, status);
    else
      gather_rows_kernel<<<AGNES_GRID(gather_rows_kernel)>>>(f, vecs, fb_id, fb_pos, total, o,
                                                             status);
  } else {
    gather_bytes_kernel<<<AGNES_GRID(gather_bytes_kernel)>>>((const uint8_t*)feats, row_bytes,
                                                             fb_id, fb_pos, total, (uint8_t*)out,
                                                             status);
  }
#undef AGNES_GRID
  return cudaGetLastError();
}

}  // namespace agnes
