// gather.cu -- feature gathering from host-resident features (staged
// blocks, the feature cache, row reads over the host link), the topology
// block loader, and the bookkeeping kernels for blocks-touched statistics.
// The gather from HBM-resident features is in gather_hbm.cu.  Every gather
// walks the final bucket, which lists each gathered node once per minibatch
// in (tile, minibatch, id) order with its output row, and copies rows as
// 16-byte vectors (bit-exact).
#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace agnes {

namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;

// Streaming variant: rows come from HBM copies of their feature blocks (a
// staging slot of the ring or the feature cache).  The batch's blocks are
// touched[0 .. nb) (ascending) and block touched[p] starts at device address
// src[p].  LPR lanes per row, each lane moving the row's 16-byte vectors
// l, l+LPR, ...
template <int LPR>
__global__ void __launch_bounds__(kThreads)
gather_staged_kernel(const unsigned long long* __restrict__ src, int64_t vecs, int64_t rpb,
                     const int32_t* __restrict__ touched, int32_t nb,
                     const int32_t* __restrict__ fb_id, const int32_t* __restrict__ fb_pos,
                     const int32_t* __restrict__ cell_off, int64_t cell_lo, int64_t cell_hi,
                     uint4* __restrict__ out, const int32_t* status) {
  grid_dep_wait();
  if (failed(status)) return;
  constexpr int kRowsPerWarp = 32 / LPR;
  const int64_t e0 = cell_off[cell_lo], e1 = cell_off[cell_hi];
  const int lane = lane_id();
  const int sub = lane / LPR, l = lane % LPR;
  const int64_t warp0 = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t i = e0 + warp0 * kRowsPerWarp + sub; i < e1; i += nwarps * kRowsPerWarp) {
    const int32_t v = __ldg(fb_id + i);
    const int64_t g = __ldg(fb_pos + i);
    const int32_t b = (int32_t)(v / rpb);
    int32_t lo = 0, hi = nb;  // position of block b in the batch
    while (hi - lo > 1) {
      const int32_t mid = (lo + hi) >> 1;
      if (__ldg(touched + mid) <= b) lo = mid; else hi = mid;
    }
    const uint4* blk = (const uint4*)__ldg(src + lo);
    const int64_t row = v - (int64_t)b * rpb;
    for (int64_t c = l; c < vecs; c += LPR)
      __stcs(out + g * vecs + c, __ldg(blk + row * vecs + c));
  }
}

// Row mode of host-resident features: every row is read from its feature
// block's current address, addr[v / rpb] -- an HBM feature-cache slot, or the
// block's pinned host memory read in place over the host link.  Walks the
// whole final bucket; LPR lanes per row, lane l moving vectors l, l+LPR, ...
// The row data is read with plain loads (it may be host memory).
template <int LPR>
__global__ void __launch_bounds__(kThreads)
gather_table_kernel(const unsigned long long* __restrict__ addr, int64_t vecs, int32_t rpb,
                    const int32_t* __restrict__ fb_id, const int32_t* __restrict__ fb_pos,
                    const int32_t* total_ptr, uint4* __restrict__ out, const int32_t* status) {
  grid_dep_wait();
  if (failed(status)) return;
  constexpr int kRowsPerWarp = 32 / LPR;
  const int64_t total = *total_ptr;
  const int lane = lane_id();
  const int sub = lane / LPR, l = lane % LPR;
  const int64_t warp0 = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t i = warp0 * kRowsPerWarp + sub; i < total; i += nwarps * kRowsPerWarp) {
    const int32_t v = __ldg(fb_id + i);
    const int64_t g = __ldg(fb_pos + i);
    const int32_t b = v / rpb;
    const uint4* src = (const uint4*)__ldg(addr + b) + (int64_t)(v - b * rpb) * vecs;
    for (int64_t c = l; c < vecs; c += LPR) __stcs(out + g * vecs + c, src[c]);
  }
}

// Copies whole feature blocks from pinned host memory, read in place over the
// host link: job j copies block blk[j] (vpb 16-byte vectors) to device address
// dst[j].  Vectors at or past host_vecs (the end of the matrix, inside its
// last block) are skipped.  The jobs form one flat range of vectors, four in
// flight per thread.
__global__ void __launch_bounds__(kThreads)
load_feat_blocks_kernel(const uint4* __restrict__ host, int64_t host_vecs,
                        const int32_t* __restrict__ blk, const unsigned long long* __restrict__ dst,
                        int32_t njobs, int64_t vpb) {
  grid_dep_wait();
  const int64_t total = (int64_t)njobs * vpb;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t q0 = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; q0 < total; q0 += 4 * stride) {
    uint4 v[4];
    int64_t j[4], r[4];
    bool ok[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int64_t q = q0 + u * stride;
      ok[u] = false;
      if (q < total) {
        j[u] = q / vpb;
        r[u] = q - j[u] * vpb;
        const int64_t s = (int64_t)__ldg(blk + j[u]) * vpb + r[u];
        if (s < host_vecs) {
          v[u] = host[s];
          ok[u] = true;
        }
      }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u)
      if (ok[u]) ((uint4*)__ldg(dst + j[u]))[r[u]] = v[u];
  }
}

__global__ void mark_kernel(const int32_t* __restrict__ cell_off, int32_t T, int32_t H,
                            const int32_t* __restrict__ map, uint8_t* __restrict__ flags,
                            const int32_t* status) {
  grid_dep_wait();
  if (failed(status)) return;
  const int64_t ncells = (int64_t)T * H;
  for (int64_t c = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; c < ncells;
       c += (int64_t)gridDim.x * blockDim.x)
    if (cell_off[c + 1] > cell_off[c]) flags[map[(uint32_t)c / (uint32_t)H]] = 1;
}

// Requests per feature block: counts[tile_feat_block[t]] += entries of tile t.
__global__ void count_requests_kernel(const int32_t* __restrict__ cell_off, int32_t T, int32_t H,
                                      const int32_t* __restrict__ tile_map,
                                      int32_t* __restrict__ counts, const int32_t* status) {
  grid_dep_wait();
  if (failed(status)) return;
  for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < T;
       t += (int64_t)gridDim.x * blockDim.x) {
    const int32_t n = cell_off[(t + 1) * H] - cell_off[t * H];
    if (n) atomicAdd(counts + tile_map[t], n);
  }
}

// Topology cache bookkeeping, per tile with frontier entries: acc[run of the
// tile] += entries, and cached += entries when the tile's block has a slot.
__global__ void count_cache_requests_kernel(const int32_t* __restrict__ cell_off, int32_t T,
                                            int32_t H, const int32_t* __restrict__ tile_adj_start,
                                            const int32_t* __restrict__ tile_adj_block,
                                            const int32_t* __restrict__ blk_slot,
                                            unsigned long long* __restrict__ acc,
                                            unsigned long long* __restrict__ cached,
                                            const int32_t* status) {
  grid_dep_wait();
  if (failed(status)) return;
  unsigned long long hit = 0;
  for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < T;
       t += (int64_t)gridDim.x * blockDim.x) {
    const int32_t n = cell_off[(t + 1) * H] - cell_off[t * H];
    if (!n) continue;
    atomicAdd(acc + tile_adj_start[t], (unsigned long long)n);
    if (blk_slot[tile_adj_block[t]] >= 0) hit += (unsigned long long)n;
  }
  hit = warp_sum(hit);
  if (lane_id() == 0 && hit) atomicAdd(cached, hit);
}

// Copies the edge lists of physical blocks from pinned host memory (read in
// place over the host link) into their graph-buffer slots: job i copies
// block jobs[i].x into slot jobs[i].y.  One CTA per job; 16-byte vectors
// where the source is aligned, single words for the ragged ends.
__global__ void __launch_bounds__(kThreads)
load_blocks_kernel(const int32_t* __restrict__ host_indices, const int64_t* __restrict__ e0,
                   const int64_t* __restrict__ e1, const int2* __restrict__ jobs, int32_t njobs,
                   int32_t* __restrict__ gbuf, int64_t epb) {
  grid_dep_wait();
  for (int32_t i = blockIdx.x; i < njobs; i += gridDim.x) {
    const int2 jb = jobs[i];
    const int64_t a = e0[jb.x], n = e1[jb.x] - a;
    const int32_t* src = host_indices + a;
    int32_t* dst = gbuf + (int64_t)jb.y * epb;
    // head words until the source is 16-byte aligned (the slot start is)
    int64_t head = (int64_t)((16 - ((uintptr_t)src & 15)) & 15) / 4;
    if (head > n) head = n;
    for (int64_t q = threadIdx.x; q < head; q += blockDim.x) dst[q] = src[q];
    const int64_t nv = (n - head) / 4;
    const int4* s4 = (const int4*)(src + head);
    for (int64_t q = threadIdx.x; q < nv; q += blockDim.x) {
      const int4 v = s4[q];
      int32_t* d = dst + head + 4 * q;  // the slot may not be 16-byte aligned here
      d[0] = v.x;
      d[1] = v.y;
      d[2] = v.z;
      d[3] = v.w;
    }
    for (int64_t q = head + 4 * nv + threadIdx.x; q < n; q += blockDim.x) dst[q] = src[q];
  }
}

// need[tile_adj_start[t]] = 1 for every tile t with a frontier entry.
__global__ void mark_runs_kernel(const int32_t* __restrict__ cell_off, int32_t T, int32_t H,
                                 const int32_t* __restrict__ tile_adj_start,
                                 uint8_t* __restrict__ need, const int32_t* status) {
  grid_dep_wait();
  if (failed(status)) return;
  for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < T;
       t += (int64_t)gridDim.x * blockDim.x)
    if (cell_off[(t + 1) * H] > cell_off[t * H]) need[tile_adj_start[t]] = 1;
}

__global__ void count_flags_kernel(const uint8_t* __restrict__ flags, int64_t n,
                                   int64_t* __restrict__ count) {
  grid_dep_wait();
  int64_t local = 0;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x)
    local += flags[i] != 0;
  local = warp_sum(local);
  if (lane_id() == 0 && local) atomicAdd((unsigned long long*)count, (unsigned long long)local);
}

// One warp per tile: union of the tile's cells over all minibatches.
__global__ void __launch_bounds__(kThreads)
distinct_rows_kernel(const int32_t* __restrict__ fb_id, const int32_t* __restrict__ cell_off,
                     const int32_t* __restrict__ tile_first, int32_t T, int32_t H,
                     unsigned long long* count) {
  grid_dep_wait();
  __shared__ uint32_t bits_s[kWarps][kTileWords];
  const int warp = threadIdx.x >> 5, lane = lane_id();
  uint32_t* bits = bits_s[warp];
  const int64_t nwarps = (int64_t)gridDim.x * kWarps;
  for (int64_t t = blockIdx.x * (int64_t)kWarps + warp; t < T; t += nwarps) {
    const int32_t base = tile_first[t];
    const int32_t words = (tile_first[t + 1] - base + 31) >> 5;
    for (int w = lane; w < words; w += 32) bits[w] = 0;
    __syncwarp();
    const int32_t o = cell_off[t * H], e = cell_off[(t + 1) * H];
    for (int32_t i = o + lane; i < e; i += 32) {
      const int32_t lu = fb_id[i] - base;
      atomicOr(&bits[lu >> 5], 1u << (lu & 31));
    }
    __syncwarp();
    uint32_t c = 0;
    for (int w = lane; w < words; w += 32) c += __popc(bits[w]);
    c = warp_sum(c);
    if (lane == 0 && c) atomicAdd(count, (unsigned long long)c);
    __syncwarp();
  }
}

// Row mode, de-duplicated: each distinct row of the hyperbatch crosses the
// host link once.  tile_bitmap_kernel (one warp per tile) records which ids
// of the tile any minibatch requests (bits), the exclusive prefix of set bits
// per 32-id word (wpref) and the count (dcnt); after a scan of dcnt into doff,
// load_distinct_rows_kernel copies distinct row d of tile t to staging row
// doff[t] + d, and gather_staged_rows_kernel serves every request from there.
__global__ void __launch_bounds__(kThreads)
tile_bitmap_kernel(const int32_t* __restrict__ fb_id, const int32_t* __restrict__ cell_off,
                   const int32_t* __restrict__ tile_first, int32_t T, int32_t H,
                   uint32_t* __restrict__ bitmap, uint16_t* __restrict__ wpref,
                   int32_t* __restrict__ dcnt, const int32_t* status) {
  grid_dep_wait();
  if (failed(status)) return;
  __shared__ uint32_t bits_s[kWarps][kTileWords];
  const int warp = threadIdx.x >> 5, lane = lane_id();
  uint32_t* bits = bits_s[warp];
  const int64_t nwarps = (int64_t)gridDim.x * kWarps;
  for (int64_t t = blockIdx.x * (int64_t)kWarps + warp; t < T; t += nwarps) {
    const int32_t base = tile_first[t];
    for (int w = lane; w < kTileWords; w += 32) bits[w] = 0;
    __syncwarp();
    const int32_t o = cell_off[t * H], e = cell_off[(t + 1) * H];
    for (int32_t i = o + lane; i < e; i += 32) {
      const int32_t lu = fb_id[i] - base;
      atomicOr(&bits[lu >> 5], 1u << (lu & 31));
    }
    __syncwarp();
    // lane l owns words 4l .. 4l+3
    uint32_t wv[4];
    int cnt = 0;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      wv[q] = bits[lane * 4 + q];
      cnt += __popc(wv[q]);
    }
    int run = warp_incl_scan(cnt) - cnt;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      bitmap[t * kTileWords + lane * 4 + q] = wv[q];
      wpref[t * kTileWords + lane * 4 + q] = (uint16_t)run;
      run += __popc(wv[q]);
    }
    if (lane == 31) dcnt[t] = run;
    __syncwarp();
  }
}

// Rank of id (in tile t, base = tile_first[t]) among the tile's requested ids.
__device__ __forceinline__ int32_t tile_rank(const uint32_t* __restrict__ bitmap,
                                             const uint16_t* __restrict__ wpref, int64_t t,
                                             int32_t lu) {
  const int64_t w = t * kTileWords + (lu >> 5);
  return (int32_t)__ldg(wpref + w) + __popc(__ldg(bitmap + w) & ((1u << (lu & 31)) - 1u));
}

// Distinct rows d of tiles [t_lo, t_hi) (d in [doff[t_lo], doff[t_hi])):
// tile t = last with doff[t] <= d; the row is the (d - doff[t])-th requested
// id of the tile, copied from its feature block's address in host memory
// (over the link; counted in *host_rows) to staging row d.  Rows of blocks in
// the feature cache, [cache_lo, cache_hi), are not staged: the gather reads
// them in place.  LPR lanes per row.
template <int LPR>
__global__ void __launch_bounds__(kThreads)
load_distinct_rows_kernel(const unsigned long long* __restrict__ addr, int64_t vecs, int32_t rpb,
                          const uint32_t* __restrict__ bitmap, const uint16_t* __restrict__ wpref,
                          const int32_t* __restrict__ doff, int32_t t_lo, int32_t t_hi,
                          const int32_t* __restrict__ tile_first, uint4* __restrict__ staging,
                          unsigned long long cache_lo, unsigned long long cache_hi,
                          unsigned long long* host_rows, const int32_t* status) {
  grid_dep_wait();
  if (failed(status)) return;
  constexpr int kRowsPerWarp = 32 / LPR;
  const int64_t d_lo = __ldg(doff + t_lo), d_hi = __ldg(doff + t_hi);
  const int lane = lane_id();
  const int sub = lane / LPR, l = lane % LPR;
  const int64_t warp0 = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  uint32_t from_host = 0;
  for (int64_t d = d_lo + warp0 * kRowsPerWarp + sub; d < d_hi; d += nwarps * kRowsPerWarp) {
    int32_t lo = t_lo, hi = t_hi;  // tile: last t with doff[t] <= d
    while (hi - lo > 1) {
      const int32_t mid = (lo + hi) >> 1;
      if (__ldg(doff + mid) <= d) lo = mid; else hi = mid;
    }
    const int32_t t = lo, r = (int32_t)(d - __ldg(doff + t));
    int32_t wl = 0, wh = kTileWords;  // word: last w with wpref[w] <= r
    while (wh - wl > 1) {
      const int32_t mid = (wl + wh) >> 1;
      if ((int32_t)__ldg(wpref + (int64_t)t * kTileWords + mid) <= r) wl = mid; else wh = mid;
    }
    const uint32_t bits = __ldg(bitmap + (int64_t)t * kTileWords + wl);
    const int32_t k = r - (int32_t)__ldg(wpref + (int64_t)t * kTileWords + wl);
    const int32_t id = __ldg(tile_first + t) + wl * 32 + (int32_t)__fns(bits, 0, k + 1);
    const int32_t b = id / rpb;
    const unsigned long long a = __ldg(addr + b);
    if (a >= cache_lo && a < cache_hi) continue;
    const uint4* src = (const uint4*)a + (int64_t)(id - b * rpb) * vecs;
    for (int64_t c = l; c < vecs; c += LPR) staging[d * vecs + c] = src[c];
    if (l == 0) ++from_host;
  }
  from_host = warp_sum(from_host);
  if (lane == 0 && from_host) atomicAdd(host_rows, (unsigned long long)from_host);
}

// Source of row id: in place in the feature cache when its block is there,
// else its staging row.
__device__ __forceinline__ const uint4* staged_row_src(
    const uint4* __restrict__ staging, int64_t vecs, const unsigned long long* __restrict__ addr,
    int32_t rpb, unsigned long long cache_lo, unsigned long long cache_hi, TileMap tm,
    const uint32_t* __restrict__ bitmap, const uint16_t* __restrict__ wpref,
    const int32_t* __restrict__ doff, int32_t id) {
  const int32_t b = id / rpb;
  const unsigned long long a = __ldg(addr + b);
  if (a >= cache_lo && a < cache_hi) return (const uint4*)a + (int64_t)(id - b * rpb) * vecs;
  const int32_t t = tile_of(tm, id);
  const int64_t srow =
      (int64_t)__ldg(doff + t) + tile_rank(bitmap, wpref, t, id - __ldg(tm.tile_first + t));
  return staging + srow * vecs;
}

// Every entry of the final bucket from the staging row of its id (or the
// feature cache).
template <int LPR, int U>
__global__ void __launch_bounds__(kThreads)
gather_staged_rows_kernel(const uint4* __restrict__ staging, const int32_t* __restrict__ fb_id,
                          const int32_t* __restrict__ fb_pos, const int32_t* lo_ptr,
                          const int32_t* hi_ptr,
                          TileMap tm, const uint32_t* __restrict__ bitmap,
                          const uint16_t* __restrict__ wpref, const int32_t* __restrict__ doff,
                          const unsigned long long* __restrict__ addr, int32_t rpb,
                          unsigned long long cache_lo, unsigned long long cache_hi,
                          uint4* __restrict__ out, const int32_t* status) {
  grid_dep_wait();
  if (failed(status)) return;
  constexpr int kRowsPerWarp = 32 / LPR;
  constexpr int kStep = kRowsPerWarp * U;
  const int64_t total = *hi_ptr;
  const int lane = lane_id();
  const int sub = lane / LPR, l = lane % LPR;
  const int64_t warp0 = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t r0 = *lo_ptr + warp0 * kStep; r0 < total; r0 += nwarps * kStep) {
    uint4 v[U];
    int32_t g[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t i = r0 + u * kRowsPerWarp + sub;
      g[u] = -1;
      if (i < total) {
        const int32_t id = __ldg(fb_id + i);
        g[u] = __ldg(fb_pos + i);
        v[u] = __ldg(staged_row_src(staging, LPR, addr, rpb, cache_lo, cache_hi, tm, bitmap, wpref,
                                    doff, id) +
                     l);
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u)
      if (g[u] >= 0) __stcs(out + (int64_t)g[u] * LPR + l, v[u]);
  }
}

// Rows of any multiple of 16 bytes: one warp per row.
__global__ void __launch_bounds__(kThreads)
gather_staged_rows_wide_kernel(const uint4* __restrict__ staging, int64_t vecs,
                               const int32_t* __restrict__ fb_id,
                               const int32_t* __restrict__ fb_pos, const int32_t* lo_ptr,
                               const int32_t* hi_ptr, TileMap tm,
                               const uint32_t* __restrict__ bitmap,
                               const uint16_t* __restrict__ wpref,
                               const int32_t* __restrict__ doff,
                               const unsigned long long* __restrict__ addr, int32_t rpb,
                               unsigned long long cache_lo, unsigned long long cache_hi,
                               uint4* __restrict__ out, const int32_t* status) {
  grid_dep_wait();
  if (failed(status)) return;
  const int64_t total = *hi_ptr;
  const int lane = lane_id();
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t i = *lo_ptr + ((blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5); i < total;
       i += nwarps) {
    const int32_t id = __ldg(fb_id + i);
    const int64_t g = __ldg(fb_pos + i);
    const uint4* src = staged_row_src(staging, vecs, addr, rpb, cache_lo, cache_hi, tm, bitmap,
                                      wpref, doff, id);
    for (int64_t c = lane; c < vecs; c += 32) __stcs(out + g * vecs + c, __ldg(src + c));
  }
}

}  // namespace

cudaError_t launch_gather_staged(const unsigned long long* src, int64_t row_bytes, int64_t rpb,
                                 const int32_t* touched, int32_t nb, const int32_t* fb_id,
                                 const int32_t* fb_pos, const int32_t* cell_off, int64_t cell_lo,
                                 int64_t cell_hi, void* out, const int32_t* status, int num_sms,
                                 cudaStream_t st) {
  const int64_t vecs = row_bytes / 16;
  uint4* o = (uint4*)out;
  // four CTAs per SM, so the block loader on the copy stream can run beside it
#define AGNES_STAGED(LPR)                                                                   \
  gather_staged_kernel<LPR><<<num_sms * 4, kThreads, 0, st>>>(src, vecs, rpb, touched, nb,   \
                                                               fb_id, fb_pos, cell_off, cell_lo, \
                                                               cell_hi, o, status)
  if (vecs <= 8)
    AGNES_STAGED(8);
  else if (vecs <= 16)
    AGNES_STAGED(16);
  else
    AGNES_STAGED(32);
#undef AGNES_STAGED
  return cudaGetLastError();
}

cudaError_t launch_gather_table(const unsigned long long* addr, int64_t row_bytes, int64_t rpb,
                                const int32_t* fb_id, const int32_t* fb_pos, const int32_t* total,
                                void* out, const int32_t* status, int num_sms, cudaStream_t st) {
  const int64_t vecs = row_bytes / 16;
  uint4* o = (uint4*)out;
#define AGNES_TABLE(LPR)                                                                    \
  gather_table_kernel<LPR><<<resident_grid((const void*)gather_table_kernel<LPR>, kThreads,  \
                                           num_sms),                                        \
                             kThreads, 0, st>>>(addr, vecs, (int32_t)rpb, fb_id, fb_pos, total, \
                                                o, status)
  if (vecs <= 8)
    AGNES_TABLE(8);
  else if (vecs <= 16)
    AGNES_TABLE(16);
  else
    AGNES_TABLE(32);
#undef AGNES_TABLE
  return cudaGetLastError();
}

cudaError_t launch_load_feat_blocks(const void* host_dev, int64_t host_bytes, const int32_t* blk,
                                    const unsigned long long* dst, int32_t njobs,
                                    int64_t block_bytes, int num_sms, cudaStream_t st) {
  if (njobs <= 0) return cudaSuccess;
  load_feat_blocks_kernel<<<num_sms, kThreads, 0, st>>>((const uint4*)host_dev, host_bytes / 16,
                                                        blk, dst, njobs, block_bytes / 16);
  return cudaGetLastError();
}

cudaError_t launch_tile_bitmaps(const int32_t* fb_id, const int32_t* cell_off,
                                const int32_t* tile_first, int32_t T, int32_t H, uint32_t* bitmap,
                                uint16_t* wpref, int32_t* dcnt, const int32_t* status,
                                cudaStream_t st) {
  tile_bitmap_kernel<<<1184, kThreads, 0, st>>>(fb_id, cell_off, tile_first, T, H, bitmap, wpref,
                                                dcnt, status);
  return cudaGetLastError();
}

cudaError_t launch_load_distinct_rows(const unsigned long long* addr, int64_t row_bytes,
                                      int64_t rpb, const uint32_t* bitmap, const uint16_t* wpref,
                                      const int32_t* doff, int32_t t_lo, int32_t t_hi,
                                      const int32_t* tile_first, void* staging,
                                      unsigned long long cache_lo, unsigned long long cache_hi,
                                      unsigned long long* host_rows, const int32_t* status,
                                      int max_blocks, int num_sms, cudaStream_t st) {
  const int64_t vecs = row_bytes / 16;
  uint4* sg = (uint4*)staging;
  if (t_hi <= t_lo) return cudaSuccess;
#define AGNES_LOADD(LPR)                                                                      \
  load_distinct_rows_kernel<LPR><<<std::min(max_blocks, resident_grid(                        \
                                       (const void*)load_distinct_rows_kernel<LPR>, kThreads,  \
                                       num_sms)),                                              \
                                   kThreads, 0, st>>>(addr, vecs, (int32_t)rpb, bitmap, wpref, \
                                                      doff, t_lo, t_hi, tile_first, sg,        \
                                                      cache_lo, cache_hi, host_rows, status)
  if (vecs <= 8)
    AGNES_LOADD(8);
  else if (vecs <= 16)
    AGNES_LOADD(16);
  else
    AGNES_LOADD(32);
#undef AGNES_LOADD
  return cudaGetLastError();
}

cudaError_t launch_gather_staged_rows(const void* staging, int64_t row_bytes, const int32_t* fb_id,
                                      const int32_t* fb_pos, const int32_t* lo, const int32_t* hi,
                                      const int32_t* tile_first, const int32_t* chunk_tile,
                                      int32_t T, const uint32_t* bitmap, const uint16_t* wpref,
                                      const int32_t* doff, const unsigned long long* addr,
                                      int64_t rpb, unsigned long long cache_lo,
                                      unsigned long long cache_hi, void* out,
                                      const int32_t* status, int num_sms, cudaStream_t st) {
  const int64_t vecs = row_bytes / 16;
  const uint4* sg = (const uint4*)staging;
  uint4* o = (uint4*)out;
  const TileMap tm{tile_first, chunk_tile, T};
#define AGNES_GSR(LPR)                                                                          \
  gather_staged_rows_kernel<LPR, 4><<<resident_grid(                                            \
                                          (const void*)gather_staged_rows_kernel<LPR, 4>,        \
                                          kThreads, num_sms),                                   \
                                      kThreads, 0, st>>>(sg, fb_id, fb_pos, lo, hi, tm, bitmap, \
                                                         wpref, doff, addr, (int32_t)rpb,       \
                                                         cache_lo, cache_hi, o, status)
  if (vecs == 8)
    AGNES_GSR(8);
  else if (vecs == 16)
    AGNES_GSR(16);
  else if (vecs == 32)
    AGNES_GSR(32);
  else
    gather_staged_rows_wide_kernel<<<resident_grid((const void*)gather_staged_rows_wide_kernel,
                                                   kThreads, num_sms),
                                     kThreads, 0, st>>>(sg, vecs, fb_id, fb_pos, lo, hi, tm, bitmap,
                                                        wpref, doff, addr, (int32_t)rpb, cache_lo,
                                                        cache_hi, o, status);
#undef AGNES_GSR
  return cudaGetLastError();
}

cudaError_t launch_mark_count(const int32_t* cell_off, int32_t T, int32_t H, const int32_t* map,
                              uint8_t* flags, int64_t n_flags, int64_t* count,
                              const int32_t* status, cudaStream_t st) {
  if (cell_off && map)
    mark_kernel<<<1184, 256, 0, st>>>(cell_off, T, H, map, flags, status);
  count_flags_kernel<<<256, 256, 0, st>>>(flags, n_flags, count);
  return cudaGetLastError();
}

cudaError_t launch_count_requests(const int32_t* cell_off, int32_t T, int32_t H,
                                  const int32_t* tile_map, int32_t* counts, int64_t n,
                                  bool zero_first, const int32_t* status, cudaStream_t st) {
  if (zero_first) {
    const cudaError_t e = cudaMemsetAsync(counts, 0, sizeof(int32_t) * (size_t)n, st);
    if (e != cudaSuccess) return e;
  }
  count_requests_kernel<<<1184, 256, 0, st>>>(cell_off, T, H, tile_map, counts, status);
  return cudaGetLastError();
}

cudaError_t launch_count_cache_requests(const int32_t* cell_off, int32_t T, int32_t H,
                                        const int32_t* tile_adj_start,
                                        const int32_t* tile_adj_block, const int32_t* blk_slot,
                                        unsigned long long* acc, unsigned long long* cached,
                                        const int32_t* status, cudaStream_t st) {
  count_cache_requests_kernel<<<1184, 256, 0, st>>>(cell_off, T, H, tile_adj_start,
                                                    tile_adj_block, blk_slot, acc, cached, status);
  return cudaGetLastError();
}

cudaError_t launch_load_blocks(const int32_t* host_indices, const int64_t* e0, const int64_t* e1,
                               const int2* jobs, int32_t njobs, int32_t* gbuf, int64_t epb,
                               int num_sms, cudaStream_t st) {
  if (njobs <= 0) return cudaSuccess;
  const int grid = njobs < num_sms * 4 ? njobs : num_sms * 4;
  load_blocks_kernel<<<grid, kThreads, 0, st>>>(host_indices, e0, e1, jobs, njobs, gbuf, epb);
  return cudaGetLastError();
}

cudaError_t launch_mark_runs(const int32_t* cell_off, int32_t T, int32_t H,
                             const int32_t* tile_adj_start, uint8_t* need, int64_t n_runs,
                             const int32_t* status, cudaStream_t st) {
  cudaError_t e = cudaMemsetAsync(need, 0, (size_t)n_runs, st);
  if (e != cudaSuccess) return e;
  mark_runs_kernel<<<1184, 256, 0, st>>>(cell_off, T, H, tile_adj_start, need, status);
  return cudaGetLastError();
}

cudaError_t launch_distinct_rows(const int32_t* fb_id, const int32_t* cell_off,
                                 const int32_t* tile_first, int32_t T, int32_t H,
                                 unsigned long long* count, cudaStream_t st) {
  distinct_rows_kernel<<<1184, kThreads, 0, st>>>(fb_id, cell_off, tile_first, T, H, count);
  return cudaGetLastError();
}

}  // namespace agnes
