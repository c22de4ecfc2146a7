// scan.cu -- segmented exclusive scans (reduce / scan-of-partials / downsweep).
//
// Used for every prefix sum on the path: the per-minibatch indptr of a hop,
// the cell offsets of the bucket matrix, the per-minibatch offsets of the new
// nodes of each (tile, minibatch) cell, and the tile compaction at load time.
// Three launches per scan and no inter-block waiting, so no kernel ever spins
// on another block's progress.
#include <mutex>
#include <unordered_map>

#include "common.cuh"
#include "internal.h"

namespace agnes {

namespace {

constexpr int kThreads = 256;
constexpr int kItems = 8;
constexpr int kChunk = kThreads * kItems;  // elements per block and chunk
// Scratch layout shared by every scan: one ticket per segment (at most
// kMaxSegments) first, kept at zero between scans, then the chunk sums.
constexpr int64_t kMaxSegments = 65536;
constexpr int64_t kTicketElems = kMaxSegments / 2;  // int64 slots holding the uint32 tickets
constexpr int64_t kGridBlocks = 2048;  // blocks of a segmented scan (at least one per segment)

__device__ __forceinline__ int64_t seg_len(const int32_t* d_len, int64_t const_len, int s) {
  return d_len ? (int64_t)d_len[s] : const_len;
}

// Exclusive block-wide scan of one int64 per thread; *total gets the sum.
__device__ __forceinline__ int64_t block_excl_scan(int64_t v, int64_t* total) {
  __shared__ int64_t warp_tot[kThreads / 32];
  __shared__ int64_t block_tot;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t incl = warp_incl_scan(v);
  if (lane == 31) warp_tot[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    const int64_t w = lane < kThreads / 32 ? warp_tot[lane] : 0;
    const int64_t wi = warp_incl_scan(w);
    if (lane < kThreads / 32) warp_tot[lane] = wi - w;
    if (lane == kThreads / 32 - 1) block_tot = wi;
  }
  __syncthreads();
  const int64_t out = warp_tot[warp] + incl - v;
  *total = block_tot;
  __syncthreads();  // warp_tot / block_tot are reused by the next call
  return out;
}

// In-place exclusive scan of n int64 values at p (element i at p[i * stride])
// by one CTA: each pass loads kItems consecutive values per thread before
// scanning them, so a pass costs one memory round trip.  Returns the total.
__device__ __forceinline__ int64_t cta_scan_inplace(int64_t* p, int64_t n, int64_t stride,
                                                   bool volatile_loads) {
  int64_t carry = 0;
  for (int64_t base = 0; base < n; base += (int64_t)kThreads * kItems) {
    const int64_t i0 = base + (int64_t)threadIdx.x * kItems;
    int64_t v[kItems];
#pragma unroll
    for (int k = 0; k < kItems; ++k) {
      const int64_t i = i0 + k;
      v[k] = i < n ? (volatile_loads ? *(volatile int64_t*)(p + i * stride) : p[i * stride]) : 0;
    }
    int64_t run = 0;
#pragma unroll
    for (int k = 0; k < kItems; ++k) {
      const int64_t x = v[k];
      v[k] = run;
      run += x;
    }
    int64_t tot;
    const int64_t ex = block_excl_scan(run, &tot);
#pragma unroll
    for (int k = 0; k < kItems; ++k) {
      const int64_t i = i0 + k;
      if (i < n) p[i * stride] = carry + ex + v[k];
    }
    carry += tot;
  }
  return carry;
}

// Chunk sums; the last chunk of a segment to finish (atomic ticket after a
// fence, no waiting) then scans the segment's chunk sums in place, writes
// the segment total, and resets the ticket for the next scan.  Only the
// chunks that hold elements of the segment take part (at least one, which
// writes the total of an empty segment); a block takes chunks blockIdx.x,
// blockIdx.x + gridDim.x, ... so the grid need not cover a segment's whole
// capacity.
template <typename InT, typename OutT>
__global__ void __launch_bounds__(kThreads)
scan_reduce_kernel(const InT* __restrict__ in, int64_t in_stride, const int32_t* d_len,
                   int64_t const_len, int64_t chunks, int64_t* __restrict__ partial,
                   unsigned int* __restrict__ tickets, OutT* __restrict__ out, int64_t out_stride,
                   bool write_end, int32_t* seg_total, const int32_t* status) {
  grid_dep_wait();
  if (status && failed(status)) return;
  const int s = blockIdx.y;
  const int64_t len = seg_len(d_len, const_len, s);
  int64_t nvalid = len > 0 ? (len + kChunk - 1) / kChunk : 1;
  if (nvalid > chunks) nvalid = chunks;
  __shared__ int64_t wsum[kThreads / 32];
  __shared__ bool last;
  for (int64_t c = blockIdx.x; c < nvalid; c += gridDim.x) {
    const int64_t begin = c * kChunk;
    int64_t sum = 0;
    if (begin < len) {  // all of the thread's loads in flight at once
      const InT* p = in + (int64_t)s * in_stride;
      InT v[kItems];
#pragma unroll
      for (int k = 0; k < kItems; ++k) {
        const int64_t i = begin + k * kThreads + threadIdx.x;
        v[k] = i < len ? p[i] : (InT)0;
      }
#pragma unroll
      for (int k = 0; k < kItems; ++k) sum += (int64_t)v[k];
    }
    sum = warp_sum(sum);
    if ((threadIdx.x & 31) == 0) wsum[threadIdx.x >> 5] = sum;
    __syncthreads();
    if (threadIdx.x < 32) {
      int64_t v = threadIdx.x < kThreads / 32 ? wsum[threadIdx.x] : 0;
      v = warp_sum(v);
      if (threadIdx.x == 0) {
        partial[(int64_t)s * chunks + c] = v;
        __threadfence();
        last = atomicAdd(tickets + s, 1u) == (unsigned)(nvalid - 1);
      }
    }
    __syncthreads();
    if (last) {  // the segment's final chunk: no later chunk of this block remains
      __threadfence();
      const int64_t carry = cta_scan_inplace(partial + (int64_t)s * chunks, nvalid, 1, true);
      if (threadIdx.x == 0) {
        if (write_end) out[(int64_t)s * out_stride + len] = (OutT)carry;
        if (seg_total) seg_total[s] = (int32_t)carry;
        tickets[s] = 0;
      }
    }
    __syncthreads();  // wsum and last are rewritten by the next chunk
  }
}

// Each warp scans 256 consecutive elements as 8 coalesced 32-wide slices
// (carry passed slice to slice), then the warps' totals are scanned.
template <typename InT, typename OutT>
__global__ void __launch_bounds__(kThreads)
scan_down_kernel(const InT* __restrict__ in, int64_t in_stride, OutT* __restrict__ out,
                 int64_t out_stride, const int32_t* d_len, int64_t const_len, int64_t chunks,
                 const int64_t* __restrict__ partial, const int32_t* status) {
  grid_dep_wait();
  if (status && failed(status)) return;
  const int s = blockIdx.y;
  const int64_t len = seg_len(d_len, const_len, s);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const InT* p = in + (int64_t)s * in_stride;
  OutT* q = out + (int64_t)s * out_stride;
  __shared__ int64_t wtot[kThreads / 32];
  for (int64_t c = blockIdx.x; c * kChunk < len; c += gridDim.x) {
    const int64_t wbase = c * kChunk + (int64_t)warp * (32 * kItems);
    const int64_t chunk_off = partial[(int64_t)s * chunks + c];  // issued with the loads below
    int64_t v[kItems];
#pragma unroll
    for (int k = 0; k < kItems; ++k) {
      const int64_t i = wbase + k * 32 + lane;
      v[k] = i < len ? (int64_t)p[i] : 0;
    }
    int64_t carry = 0;
#pragma unroll
    for (int k = 0; k < kItems; ++k) {
      const int64_t inc = warp_incl_scan(v[k]);
      const int64_t x = v[k];
      v[k] = carry + inc - x;
      carry += __shfl_sync(0xffffffffu, inc, 31);
    }
    if (lane == 0) wtot[warp] = carry;
    __syncthreads();
    if (warp == 0) {
      const int64_t w = lane < kThreads / 32 ? wtot[lane] : 0;
      const int64_t wi = warp_incl_scan(w);
      if (lane < kThreads / 32) wtot[lane] = wi - w;
    }
    __syncthreads();
    const int64_t off = chunk_off + wtot[warp];
#pragma unroll
    for (int k = 0; k < kItems; ++k) {
      const int64_t i = wbase + k * 32 + lane;
      if (i < len) q[i] = (OutT)(off + v[k]);
    }
    __syncthreads();  // wtot is rewritten by the next chunk
  }
}

// ---- column scan of a row-major [rows x cols] matrix ----------------------------
constexpr int kColRows = 16;  // rows per chunk

__global__ void __launch_bounds__(128)
col_reduce_kernel(const int32_t* __restrict__ in, int64_t rows, int32_t cols,
                  int64_t* __restrict__ partial, const int32_t* status) {
  grid_dep_wait();
  if (status && failed(status)) return;
  const int32_t c = blockIdx.y * 128 + threadIdx.x;
  if (c >= cols) return;
  const int64_t r0 = (int64_t)blockIdx.x * kColRows;
  const int64_t r1 = min(rows, r0 + kColRows);
  int32_t v[kColRows];
#pragma unroll
  for (int k = 0; k < kColRows; ++k) v[k] = r0 + k < r1 ? in[(r0 + k) * cols + c] : 0;
  int64_t sum = 0;
#pragma unroll
  for (int k = 0; k < kColRows; ++k) sum += v[k];
  partial[(int64_t)blockIdx.x * cols + c] = sum;
}

// One CTA per column: exclusive scan of its chunk partials (strided by cols).
__global__ void __launch_bounds__(kThreads)
col_partials_kernel(int64_t* __restrict__ partial, int64_t chunks, int32_t cols,
                    const int32_t* __restrict__ add_in, int32_t* __restrict__ total_out,
                    const int32_t* status) {
  grid_dep_wait();
  if (status && failed(status)) return;
  const int32_t c = blockIdx.x;
  const int64_t carry = cta_scan_inplace(partial + c, chunks, cols, false);
  if (threadIdx.x == 0 && total_out)
    total_out[c] = (int32_t)carry + (add_in ? add_in[c] : 0);
}

__global__ void __launch_bounds__(128)
col_down_kernel(const int32_t* __restrict__ in, int32_t* __restrict__ out, int64_t rows,
                int32_t cols, const int64_t* __restrict__ partial, const int32_t* status) {
  grid_dep_wait();
  if (status && failed(status)) return;
  const int32_t c = blockIdx.y * 128 + threadIdx.x;
  if (c >= cols) return;
  const int64_t r0 = (int64_t)blockIdx.x * kColRows;
  const int64_t r1 = min(rows, r0 + kColRows);
  int64_t run = partial[(int64_t)blockIdx.x * cols + c];
  int32_t v[kColRows];
#pragma unroll
  for (int k = 0; k < kColRows; ++k) v[k] = r0 + k < r1 ? in[(r0 + k) * cols + c] : 0;
#pragma unroll
  for (int k = 0; k < kColRows; ++k) {
    if (r0 + k < r1) out[(r0 + k) * cols + c] = (int32_t)run;
    run += v[k];
  }
}

// ---- single-pass flat scan (decoupled look-back) ----------------------------------
//
// Merrill & Garland's single-pass prefix scan (2016): every CTA takes the next
// tile of kFlatTile elements from a counter, publishes its tile's sum, and
// derives its exclusive prefix by walking back over its predecessors' flags
// until it meets an inclusive prefix; it then publishes that as well.  CTAs
// take tiles in the order they start, so a CTA waits only on tiles of CTAs
// that are already running; each wait is still bounded (kFlatSpinLimit
// polls), after which the CTA records kErrWaitTimeout and carries on.
//
// Scratch (uint64, zero between scans): [0] tile counter, [1] finished
// CTAs, [2 + t] flag of tile t = state << 62 | value, state 1 = the tile's
// sum, 2 = the inclusive prefix through the tile.  The last CTA to finish
// clears the flags and the counters.
constexpr int kFlatItems = 16;  // consecutive elements per thread (four 16-byte vectors)
constexpr int64_t kFlatTile = (int64_t)kThreads * kFlatItems;
constexpr unsigned long long kFlagAgg = 1ull << 62;
constexpr unsigned long long kFlagInc = 2ull << 62;
constexpr unsigned long long kFlagVal = (1ull << 62) - 1;
constexpr int kFlatSpinLimit = 1 << 20;

__device__ __forceinline__ unsigned long long flag_load(const unsigned long long* p) {
  return *(const volatile unsigned long long*)p;
}

__global__ void __launch_bounds__(kThreads)
flat_scan_kernel(const int32_t* __restrict__ in, int32_t* __restrict__ out, int64_t n,
                 bool write_end, int32_t* total_out, unsigned long long* scratch,
                 int32_t* status) {
  grid_dep_wait();
  // no early return on a failed status: every CTA takes its tile and counts
  // itself finished, so the scratch is left zero for the next scan
  __shared__ int64_t s_tile, s_excl;
  __shared__ int64_t warp_tot[kThreads / 32];
  __shared__ bool s_last;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t ntiles = (int64_t)gridDim.x;
  unsigned long long* flags = scratch + 2;
  if (tid == 0) {
    const int64_t t = (int64_t)atomicAdd(scratch, 1ull);
    if (t == ntiles - 1) scratch[0] = 0;  // every CTA has taken its tile
    s_tile = t;
  }
  __syncthreads();
  const int64_t tile = s_tile;
  // the thread's 16 consecutive elements
  const int64_t i0 = tile * kFlatTile + (int64_t)tid * kFlatItems;
  int32_t v[kFlatItems];
  if (i0 + kFlatItems <= n) {
    const int4* p = reinterpret_cast<const int4*>(in + i0);
#pragma unroll
    for (int q = 0; q < kFlatItems / 4; ++q) {
      const int4 x = p[q];
      v[4 * q] = x.x;
      v[4 * q + 1] = x.y;
      v[4 * q + 2] = x.z;
      v[4 * q + 3] = x.w;
    }
  } else {
#pragma unroll
    for (int k = 0; k < kFlatItems; ++k) v[k] = i0 + k < n ? in[i0 + k] : 0;
  }
  int64_t mine = 0;
#pragma unroll
  for (int k = 0; k < kFlatItems; ++k) mine += v[k];
  // block scan of the threads' sums
  const int64_t incl = warp_incl_scan(mine);
  if (lane == 31) warp_tot[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    const int64_t w = lane < kThreads / 32 ? warp_tot[lane] : 0;
    const int64_t wi = warp_incl_scan(w);
    if (lane < kThreads / 32) warp_tot[lane] = wi - w;
    const int64_t agg = __shfl_sync(0xffffffffu, wi, kThreads / 32 - 1);
    // publish, look back, publish the inclusive prefix
    int64_t excl = 0;
    if (tile == 0) {
      if (lane == 0) atomicExch(flags, kFlagInc | (unsigned long long)agg);
    } else {
      if (lane == 0) atomicExch(flags + tile, kFlagAgg | (unsigned long long)agg);
      for (int64_t j = tile - 1;; j -= 32) {
        const int64_t idx = j - lane;  // lane 0 the nearest predecessor
        unsigned long long f = kFlagInc;  // before tile 0: an inclusive prefix of 0
        if (idx >= 0) {
          f = flag_load(flags + idx);
          for (int spin = 0; (f >> 62) == 0; ++spin) {
            if (spin == kFlatSpinLimit) {
              atomicOr(status, kErrWaitTimeout);
              f = kFlagInc;
              break;
            }
            __nanosleep(64);
            f = flag_load(flags + idx);
          }
        }
        const unsigned inc = __ballot_sync(0xffffffffu, (f >> 62) == 2);
        const int stop = inc ? __ffs(inc) - 1 : 31;  // lanes 0 .. stop contribute
        excl += warp_sum(lane <= stop ? (int64_t)(f & kFlagVal) : (int64_t)0);
        if (inc) break;
      }
      if (lane == 0) atomicExch(flags + tile, kFlagInc | (unsigned long long)(excl + agg));
    }
    if (lane == 0) {
      s_excl = excl;
      if (tile == ntiles - 1) {
        if (write_end) out[n] = (int32_t)(excl + agg);
        if (total_out) *total_out = (int32_t)(excl + agg);
      }
    }
  }
  __syncthreads();
  int64_t run = s_excl + warp_tot[warp] + incl - mine;
  int32_t o[kFlatItems];
#pragma unroll
  for (int k = 0; k < kFlatItems; ++k) {
    o[k] = (int32_t)run;
    run += v[k];
  }
  if (i0 + kFlatItems <= n) {
    int4* p = reinterpret_cast<int4*>(out + i0);
#pragma unroll
    for (int q = 0; q < kFlatItems / 4; ++q)
      p[q] = make_int4(o[4 * q], o[4 * q + 1], o[4 * q + 2], o[4 * q + 3]);
  } else {
#pragma unroll
    for (int k = 0; k < kFlatItems; ++k)
      if (i0 + k < n) out[i0 + k] = o[k];
  }
  // the last CTA to finish (all look-backs done) clears the scratch
  if (tid == 0) {
    __threadfence();
    s_last = atomicAdd(scratch + 1, 1ull) == (unsigned long long)(ntiles - 1);
  }
  __syncthreads();
  if (s_last) {
    for (int64_t t = tid; t < ntiles; t += kThreads) flags[t] = 0;
    if (tid == 0) scratch[1] = 0;
  }
}

}  // namespace

int64_t col_scan_scratch_elems(int64_t rows, int32_t cols) {
  return kTicketElems + ((rows + kColRows - 1) / kColRows) * (int64_t)cols;
}

cudaError_t col_scan(const int32_t* in, int32_t* out, int64_t rows, int32_t cols,
                     const int32_t* add_in, int32_t* total_out, int64_t* scratch,
                     const int32_t* status, cudaStream_t st) {
  if (rows <= 0 || cols <= 0) return cudaSuccess;
  const int64_t chunks = (rows + kColRows - 1) / kColRows;
  const dim3 grid((unsigned)chunks, (unsigned)((cols + 127) / 128));
  int64_t* partial = scratch + kTicketElems;  // leave the seg_scan tickets untouched
  col_reduce_kernel<<<grid, 128, 0, st>>>(in, rows, cols, partial, status);
  col_partials_kernel<<<cols, kThreads, 0, st>>>(partial, chunks, cols, add_in, total_out, status);
  col_down_kernel<<<grid, 128, 0, st>>>(in, out, rows, cols, partial, status);
  return cudaGetLastError();
}

int resident_grid(const void* kernel, int threads, int num_sms) {
  static std::mutex mu;
  static std::unordered_map<const void*, int> per_sm_cache;
  int per_sm = 0;
  {
    std::lock_guard<std::mutex> lock(mu);
    auto it = per_sm_cache.find(kernel);
    if (it != per_sm_cache.end()) per_sm = it->second;
  }
  if (per_sm == 0) {
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, threads, 0) !=
            cudaSuccess ||
        per_sm < 1) {
      cudaGetLastError();
      per_sm = 1;
    }
    std::lock_guard<std::mutex> lock(mu);
    per_sm_cache[kernel] = per_sm;
  }
  return per_sm * num_sms;
}

int64_t scan_scratch_elems(int64_t nseg, int64_t max_len) {
  int64_t chunks = (max_len + kChunk - 1) / kChunk;
  if (chunks < 1) chunks = 1;
  return kTicketElems + nseg * chunks;
}

int64_t flat_scan_scratch_elems(int64_t max_n) {
  return 2 + (max_n + kFlatTile - 1) / kFlatTile + 1;
}

bool flat_scan_supported(const int32_t* in, const int32_t* out) {
  return (uintptr_t)in % 16 == 0 && (uintptr_t)out % 16 == 0;
}

cudaError_t flat_scan(const int32_t* in, int32_t* out, int64_t n, bool write_end,
                      int32_t* total_out, uint64_t* scratch, int32_t* status, cudaStream_t st) {
  if (!flat_scan_supported(in, out)) return cudaErrorInvalidValue;
  const int64_t ntiles = n > 0 ? (n + kFlatTile - 1) / kFlatTile : 1;
  if (ntiles > 0x7fffffff) return cudaErrorInvalidValue;
  flat_scan_kernel<<<(unsigned)ntiles, kThreads, 0, st>>>(
      in, out, n, write_end, total_out, reinterpret_cast<unsigned long long*>(scratch), status);
  return cudaGetLastError();
}

template <typename InT, typename OutT>
cudaError_t seg_scan(const InT* in, int64_t in_stride, OutT* out, int64_t out_stride,
                     const int32_t* d_len, int64_t const_len, int32_t nseg, int64_t max_len,
                     bool write_end, int32_t* seg_total, int64_t* scratch,
                     const int32_t* status, cudaStream_t st) {
  if (nseg <= 0) return cudaSuccess;
  int64_t chunks = (max_len + kChunk - 1) / kChunk;
  if (chunks < 1) chunks = 1;
  // Segments of a per-minibatch scan are usually far shorter than their
  // capacity max_len: about kGridBlocks blocks in all, each looping over its
  // segment's chunks, instead of a block per chunk of capacity.
  int64_t gx = kGridBlocks / nseg;
  if (gx < 1) gx = 1;
  if (gx > chunks) gx = chunks;
  const dim3 grid((unsigned)gx, (unsigned)nseg);
  if (nseg > kMaxSegments) return cudaErrorInvalidValue;
  unsigned int* tickets = (unsigned int*)scratch;
  int64_t* partial = scratch + kTicketElems;
  scan_reduce_kernel<InT, OutT><<<grid, kThreads, 0, st>>>(in, in_stride, d_len, const_len, chunks,
                                                           partial, tickets, out, out_stride,
                                                           write_end, seg_total, status);
  scan_down_kernel<InT, OutT><<<grid, kThreads, 0, st>>>(in, in_stride, out, out_stride, d_len,
                                                         const_len, chunks, partial, status);
  return cudaGetLastError();
}

template cudaError_t seg_scan<int32_t, int32_t>(const int32_t*, int64_t, int32_t*, int64_t,
                                                const int32_t*, int64_t, int32_t, int64_t, bool,
                                                int32_t*, int64_t*, const int32_t*, cudaStream_t);
template cudaError_t seg_scan<int32_t, int64_t>(const int32_t*, int64_t, int64_t*, int64_t,
                                                const int32_t*, int64_t, int32_t, int64_t, bool,
                                                int32_t*, int64_t*, const int32_t*, cudaStream_t);
template cudaError_t seg_scan<uint8_t, int32_t>(const uint8_t*, int64_t, int32_t*, int64_t,
                                                const int32_t*, int64_t, int32_t, int64_t, bool,
                                                int32_t*, int64_t*, const int32_t*, cudaStream_t);

}  // namespace agnes
