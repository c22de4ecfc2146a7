// noalloc.cu -- agnes_hop_indptr_noalloc: one hop's per-node edge counts
// min(deg(v), fanout) and their prefix sum for a caller's node list, with all
// scratch in a file-scope device array, so the call allocates nothing.
//
// It is a stand-alone variant of the count + scan step the hyperbatch path
// runs before each hop's sampling (sample.cu's count kernel and scan.cu's
// segmented scan), kept separate so that path stays as it is.
//
// Scratch: the per-chunk partial sums and an error word live in g_scratch.
// Host code may not use the name g_scratch as a device address: every call
// looks the array's address up with cudaGetSymbolAddress (with the ctx's
// device current) and every launch gets that pointer.  Every call on a device
// shares the array, so calls that overlap on the GPU race; the error word is
// cleared at the start of each call and the partial sums are fully rewritten
// by each call.
#include "../../include/agnes.h"
#include "common.cuh"
#include "internal.h"

namespace agnes {

namespace {

constexpr int kNaThreads = 256;
constexpr int kNaItems = 8;
constexpr int kNaChunk = kNaThreads * kNaItems;  // nodes per chunk
constexpr int kNaMaxChunks = (int)(AGNES_NOALLOC_MAX_NODES / kNaChunk);
constexpr int kNaErrWord = kNaMaxChunks;  // index of the error word

static_assert(AGNES_NOALLOC_MAX_NODES % kNaChunk == 0, "chunking must tile the maximum");

// chunk partial sums [0, kNaMaxChunks), error word at kNaErrWord (64 KiB)
static __device__ __align__(256) int64_t g_scratch[kNaMaxChunks + 32];

template <typename OffT>
__device__ __forceinline__ int64_t hop_count(const OffT* __restrict__ off, int64_t N,
                                             const int32_t* __restrict__ nodes, int64_t i,
                                             int32_t k, int64_t* scratch) {
  const int32_t v = nodes[i];
  if (v < 0 || v >= N) {
    atomicOr((unsigned long long*)(scratch + kNaErrWord), 1ull);
    return 0;
  }
  const int64_t d = (int64_t)off[v + 1] - (int64_t)off[v];
  return d < k ? d : k;
}

__device__ __forceinline__ int64_t na_block_excl_scan(int64_t v, int64_t* total) {
  __shared__ int64_t warp_tot[kNaThreads / 32];
  __shared__ int64_t block_tot;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t incl = warp_incl_scan(v);
  if (lane == 31) warp_tot[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    const int64_t w = lane < kNaThreads / 32 ? warp_tot[lane] : 0;
    const int64_t wi = warp_incl_scan(w);
    if (lane < kNaThreads / 32) warp_tot[lane] = wi - w;
    if (lane == kNaThreads / 32 - 1) block_tot = wi;
  }
  __syncthreads();
  const int64_t out = warp_tot[warp] + incl - v;
  *total = block_tot;
  __syncthreads();
  return out;
}

__global__ void na_clear_kernel(int64_t* scratch) { scratch[kNaErrWord] = 0; }

template <typename OffT>
__global__ void __launch_bounds__(kNaThreads)
na_reduce_kernel(const OffT* __restrict__ off, int64_t N, const int32_t* __restrict__ nodes,
                 int64_t n, int32_t k, int64_t* scratch) {
  const int64_t begin = (int64_t)blockIdx.x * kNaChunk;
  const int64_t end = min(n, begin + kNaChunk);
  int64_t sum = 0;
  for (int64_t i = begin + threadIdx.x; i < end; i += kNaThreads)
    sum += hop_count(off, N, nodes, i, k, scratch);
  int64_t tot;
  na_block_excl_scan(sum, &tot);
  if (threadIdx.x == 0) scratch[blockIdx.x] = tot;
}

__global__ void __launch_bounds__(kNaThreads)
na_partials_kernel(int64_t chunks, int64_t n, int64_t* scratch, int64_t* __restrict__ indptr) {
  int64_t carry = 0;
  for (int64_t base = 0; base < chunks; base += kNaThreads) {
    const int64_t i = base + threadIdx.x;
    const int64_t v = i < chunks ? scratch[i] : 0;
    int64_t tot;
    const int64_t ex = na_block_excl_scan(v, &tot);
    if (i < chunks) scratch[i] = carry + ex;
    carry += tot;
  }
  if (threadIdx.x == 0) indptr[n] = carry;
}

template <typename OffT>
__global__ void __launch_bounds__(kNaThreads)
na_down_kernel(const OffT* __restrict__ off, int64_t N, const int32_t* __restrict__ nodes,
               int64_t n, int32_t k, const int64_t* scratch_in, int64_t* scratch,
               int64_t* __restrict__ indptr) {
  const int64_t begin = (int64_t)blockIdx.x * kNaChunk + (int64_t)threadIdx.x * kNaItems;
  int64_t c[kNaItems];
  int64_t run = 0;
#pragma unroll
  for (int q = 0; q < kNaItems; ++q) {
    const int64_t i = begin + q;
    c[q] = i < n ? hop_count(off, N, nodes, i, k, scratch) : 0;
    run += c[q];
  }
  int64_t tot;
  int64_t ex = na_block_excl_scan(run, &tot) + scratch_in[blockIdx.x];
#pragma unroll
  for (int q = 0; q < kNaItems; ++q) {
    const int64_t i = begin + q;
    if (i < n) indptr[i] = ex;
    ex += c[q];
  }
}

// Device address of g_scratch on the current device.  Looked up on every
// call (a host-side query, no device work), so that no address outlives the
// context it was taken in: after a cudaDeviceReset the next call gets the
// array of the new context.
cudaError_t na_scratch(int64_t** out) {
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_scratch);
  if (e != cudaSuccess) return e;
  *out = (int64_t*)p;
  return cudaSuccess;
}

bool na_is_device_ptr(const void* p) {
  cudaPointerAttributes attr;
  if (cudaPointerGetAttributes(&attr, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return attr.type == cudaMemoryTypeDevice || attr.type == cudaMemoryTypeManaged;
}

}  // namespace

}  // namespace agnes

using namespace agnes;

extern "C" agnes_status agnes_hop_indptr_noalloc(agnes_ctx* ctx, const int32_t* nodes, int64_t n,
                                                 int32_t fanout, int64_t* indptr,
                                                 void* cuda_stream) {
  if (!ctx || !indptr || (n > 0 && !nodes) || n < 0) {
    ctx_set_error(ctx, "ctx, nodes and indptr must be non-NULL and n >= 0");
    return AGNES_EINVAL;
  }
  if (n > AGNES_NOALLOC_MAX_NODES) {
    ctx_set_error(ctx, "agnes_hop_indptr_noalloc takes at most %lld nodes, got %lld",
                  (long long)AGNES_NOALLOC_MAX_NODES, (long long)n);
    return AGNES_ERANGE;
  }
  if (fanout < 1 || fanout > AGNES_MAX_FANOUT) {
    ctx_set_error(ctx, "fanout %d outside [1, %d]", fanout, AGNES_MAX_FANOUT);
    return AGNES_EINVAL;
  }
  GraphView g;
  ctx_graph_view(ctx, &g);
  DeviceGuard dg(g.device);
  if (!dg.ok()) {
    ctx_set_error(ctx, "cudaSetDevice(%d) failed", g.device);
    return AGNES_ECUDA;
  }
  if (!na_is_device_ptr(indptr) || (n > 0 && !na_is_device_ptr(nodes))) {
    ctx_set_error(ctx, "nodes and indptr must be device memory");
    return AGNES_EINVAL;
  }
  int64_t* scratch = nullptr;
  cudaError_t e = na_scratch(&scratch);
  if (e != cudaSuccess) {
    ctx_set_error(ctx, "cudaGetSymbolAddress failed: %s", cudaGetErrorString(e));
    return AGNES_ECUDA;
  }
  cudaStream_t st = (cudaStream_t)cuda_stream;
  if (n == 0) {
    e = cudaMemsetAsync(indptr, 0, sizeof(int64_t), st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) {
      ctx_set_error(ctx, "%s", cudaGetErrorString(e));
      return AGNES_ECUDA;
    }
    return AGNES_OK;
  }
  const int64_t chunks = (n + kNaChunk - 1) / kNaChunk;
  na_clear_kernel<<<1, 1, 0, st>>>(scratch);
  if (g.offsets_bits == 32) {
    const int32_t* off = (const int32_t*)g.offsets;
    na_reduce_kernel<int32_t><<<(unsigned)chunks, kNaThreads, 0, st>>>(off, g.N, nodes, n, fanout,
                                                                       scratch);
    na_partials_kernel<<<1, kNaThreads, 0, st>>>(chunks, n, scratch, indptr);
    na_down_kernel<int32_t><<<(unsigned)chunks, kNaThreads, 0, st>>>(off, g.N, nodes, n, fanout,
                                                                     scratch, scratch, indptr);
  } else {
    const int64_t* off = (const int64_t*)g.offsets;
    na_reduce_kernel<int64_t><<<(unsigned)chunks, kNaThreads, 0, st>>>(off, g.N, nodes, n, fanout,
                                                                       scratch);
    na_partials_kernel<<<1, kNaThreads, 0, st>>>(chunks, n, scratch, indptr);
    na_down_kernel<int64_t><<<(unsigned)chunks, kNaThreads, 0, st>>>(off, g.N, nodes, n, fanout,
                                                                     scratch, scratch, indptr);
  }
  e = cudaGetLastError();
  int64_t err = 0;
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(&err, scratch + kNaErrWord, sizeof(err), cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) {
    ctx_set_error(ctx, "%s", cudaGetErrorString(e));
    return AGNES_ECUDA;
  }
  if (err) {
    ctx_set_error(ctx, "a node id is outside [0, %lld)", (long long)g.N);
    return AGNES_EINVAL;
  }
  return AGNES_OK;
}
