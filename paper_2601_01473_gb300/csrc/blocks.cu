// blocks.cu -- block tables built once per graph (Sec. 3.2, storage layer).
//
// Topology blocks: objects (an offset header of offsets_bits/8 bytes plus 4
// bytes per neighbour) are packed greedily in ascending node id into blocks of
// adj_block_bytes; an object that does not fit in the rest of the current
// block starts the next one; an object larger than a block starts a fresh
// block and spans ceil(size / block) blocks.  The packing is a chain (each
// block's first node depends on the previous block), so one warp walks it:
// with P(v) = v*hdr + 4*offsets[v] the byte prefix of the objects, the block
// starting at v ends before the largest w with P(w) - P(v) <= block, found by
// a 32-ary search over at most block/hdr candidates.  The result is the
// object index table T^g_obj: (first node, block index) per block start.
//
// Feature blocks: rows_per_block consecutive rows each.
//
// Tiles: the common refinement of topology blocks, feature blocks and 4096-id
// chunks.  Buckets are kept per (tile, minibatch) cell; a tile maps to exactly
// one topology block and one feature block.
#include <stdio.h>

#include "common.cuh"
#include "internal.h"

namespace agnes {

namespace {

template <typename OffT>
__device__ __forceinline__ int64_t obj_prefix(const OffT* off, int64_t v, int64_t hdr) {
  return v * hdr + 4 * (int64_t)off[v];
}

// out[0] = number of block starts, out[1] = number of blocks, out[2] = 1 when
// the start table overflowed (cannot happen with the host's bound).
template <typename OffT>
__global__ void adj_chain_kernel(const OffT* __restrict__ off, int64_t N, int64_t hdr, int64_t bb,
                                 int32_t* __restrict__ start_node, int32_t* __restrict__ start_block,
                                 int64_t cap, int64_t* out) {
  const int lane = threadIdx.x & 31;
  const int64_t max_objs = bb / hdr;
  int64_t v = 0, b = 0, n = 0, overflow = 0;
  while (v < N) {
    if (n >= cap) {
      overflow = 1;
      break;
    }
    if (lane == 0) {
      start_node[n] = (int32_t)v;
      start_block[n] = (int32_t)b;
    }
    ++n;
    const int64_t pv = obj_prefix(off, v, hdr);
    const int64_t size = obj_prefix(off, v + 1, hdr) - pv;
    if (size > bb) {
      b += (size + bb - 1) / bb;
      v += 1;
      continue;
    }
    // Largest w in [v+1, hi] with P(w) - P(v) <= bb; P(v+1) - P(v) <= bb holds.
    int64_t lo = v + 1;
    int64_t hi = min(N, v + max_objs);
    while (hi > lo) {
      const int64_t step = (hi - lo + 31) / 32;
      const int64_t p = min(hi, lo + step * (lane + 1));
      const bool ok = obj_prefix(off, p, hdr) - pv <= bb;
      const int cnt = __popc(__ballot_sync(0xffffffffu, ok));
      const int64_t nlo = cnt > 0 ? min(hi, lo + step * cnt) : lo;
      const int64_t nhi = cnt < 32 ? min(hi, lo + step * (cnt + 1)) - 1 : hi;
      lo = nlo;
      hi = nhi;
    }
    b += 1;
    v = lo;
  }
  if (lane == 0) {
    out[0] = n;
    out[1] = b;
    out[2] = overflow;
  }
}

__global__ void tile_flags_kernel(uint8_t* __restrict__ flags, int64_t N, int64_t rpb) {
  for (int64_t v = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; v < N;
       v += (int64_t)gridDim.x * blockDim.x)
    flags[v] = ((v & (kTileSpan - 1)) == 0) || (v % rpb == 0);
}

__global__ void tile_flag_starts_kernel(uint8_t* __restrict__ flags,
                                        const int32_t* __restrict__ start_node, int64_t n) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x)
    flags[start_node[i]] = 1;
}

__global__ void tile_compact_kernel(const uint8_t* __restrict__ flags,
                                    const int32_t* __restrict__ rank, int64_t N,
                                    int32_t* __restrict__ tile_first,
                                    int32_t* __restrict__ chunk_tile) {
  for (int64_t v = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; v < N;
       v += (int64_t)gridDim.x * blockDim.x) {
    if (flags[v]) {
      const int32_t t = rank[v];
      tile_first[t] = (int32_t)v;
      if ((v & (kTileSpan - 1)) == 0) chunk_tile[v >> kTileShift] = t;
    }
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    const int32_t T = rank[N];
    tile_first[T] = (int32_t)N;
    chunk_tile[(N + kTileSpan - 1) >> kTileShift] = T;
  }
}

__global__ void tile_blocks_kernel(const int32_t* __restrict__ tile_first, int64_t T,
                                   const int32_t* __restrict__ start_node,
                                   const int32_t* __restrict__ start_block, int64_t n_starts,
                                   int64_t rpb, int32_t* __restrict__ tile_adj_block,
                                   int32_t* __restrict__ tile_feat_block,
                                   int32_t* __restrict__ tile_adj_start,
                                   int32_t* __restrict__ run_first_tile) {
  for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < T;
       t += (int64_t)gridDim.x * blockDim.x) {
    const int32_t v = tile_first[t];
    // last block start <= v
    int64_t lo = 0, hi = n_starts;
    while (hi - lo > 1) {
      const int64_t mid = (lo + hi) >> 1;
      if (start_node[mid] <= v)
        lo = mid;
      else
        hi = mid;
    }
    tile_adj_block[t] = start_block[lo];
    tile_feat_block[t] = (int32_t)(v / rpb);
    tile_adj_start[t] = (int32_t)lo;
    if (start_node[lo] == v) run_first_tile[lo] = (int32_t)t;  // block starts start tiles
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) run_first_tile[n_starts] = (int32_t)T;
}

// Edge range [e0, e1) of every physical block: a block of whole objects
// holds the edges of its nodes; the i-th block of an object larger than a
// block holds the edges whose bytes (after the hdr-byte header) fall in
// [i*bb, (i+1)*bb) of the object.
template <typename OffT>
__global__ void block_edges_kernel(const OffT* __restrict__ off, int64_t N, int64_t hdr, int64_t bb,
                                   const int32_t* __restrict__ start_node,
                                   const int32_t* __restrict__ start_block, int64_t n_starts,
                                   int64_t n_blocks, int64_t* __restrict__ e0,
                                   int64_t* __restrict__ e1) {
  for (int64_t s = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; s < n_starts;
       s += (int64_t)gridDim.x * blockDim.x) {
    const int64_t v0 = start_node[s];
    const int64_t v1 = s + 1 < n_starts ? start_node[s + 1] : N;
    const int64_t b0 = start_block[s];
    const int64_t b1 = s + 1 < n_starts ? start_block[s + 1] : n_blocks;
    const int64_t a = (int64_t)off[v0], z = (int64_t)off[v1];
    if (b1 - b0 == 1) {
      e0[b0] = a;
      e1[b0] = z;
    } else {  // one big object
      const int64_t deg = z - a;
      for (int64_t i = 0; i < b1 - b0; ++i) {
        int64_t lo = (i * bb - hdr + 3) / 4;
        int64_t hi = ((i + 1) * bb - hdr + 3) / 4;
        lo = lo < 0 ? 0 : (lo > deg ? deg : lo);
        hi = hi < 0 ? 0 : (hi > deg ? deg : hi);
        e0[b0 + i] = a + lo;
        e1[b0 + i] = a + hi;
      }
    }
  }
}

// First tile of each feature block (multiples of rows_per_block start tiles).
__global__ void fblock_first_tile_kernel(const int32_t* __restrict__ tile_first,
                                         const int32_t* __restrict__ tile_feat_block, int64_t T,
                                         int64_t rpb, int64_t nfb,
                                         int32_t* __restrict__ fblock_first_tile) {
  for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < T;
       t += (int64_t)gridDim.x * blockDim.x) {
    const int32_t b = tile_feat_block[t];
    if ((int64_t)tile_first[t] == (int64_t)b * rpb) fblock_first_tile[b] = (int32_t)t;
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) fblock_first_tile[nfb] = (int32_t)T;
}

}  // namespace

void free_block_tables(BlockTables* bt) {
  cudaFree(bt->start_node);
  cudaFree(bt->start_block);
  cudaFree(bt->tile_first);
  cudaFree(bt->chunk_tile);
  cudaFree(bt->tile_adj_block);
  cudaFree(bt->tile_feat_block);
  cudaFree(bt->fblock_first_tile);
  cudaFree(bt->tile_adj_start);
  cudaFree(bt->run_first_tile);
  cudaFree(bt->blk_e0);
  cudaFree(bt->blk_e1);
  *bt = BlockTables();
}

#define BT_CHECK(call)                                                                 \
  do {                                                                                 \
    cudaError_t e_ = (call);                                                           \
    if (e_ != cudaSuccess) {                                                           \
      snprintf(err, errlen, "%s: %s", #call, cudaGetErrorString(e_));                  \
      rc = e_;                                                                         \
      goto done;                                                                       \
    }                                                                                  \
  } while (0)

cudaError_t build_block_tables(const void* d_offsets, int offsets_bits, int64_t N, int64_t E,
                               int64_t adj_block_bytes, int64_t rows_per_feat_block,
                               BlockTables* bt, cudaStream_t st, char* err, size_t errlen) {
  cudaError_t rc = cudaSuccess;
  const int64_t hdr = offsets_bits / 8;
  const int64_t total_bytes = N * hdr + 4 * E;
  const int64_t bound = 2 * ((total_bytes + adj_block_bytes - 1) / adj_block_bytes) + 2;
  const int64_t cap = bound < N ? bound : N;
  const int64_t C = (N + kTileSpan - 1) / kTileSpan;
  int64_t host_out[3] = {0, 0, 0};
  int64_t* d_out = nullptr;
  uint8_t* flags = nullptr;
  int32_t* rank = nullptr;
  int64_t* scratch = nullptr;
  int32_t T32 = 0;
  const int grid = 1184;

  *bt = BlockTables();
  bt->rows_per_feat_block = rows_per_feat_block;
  bt->n_feat_blocks = (N + rows_per_feat_block - 1) / rows_per_feat_block;

  BT_CHECK(cudaMalloc(&bt->start_node, sizeof(int32_t) * cap));
  BT_CHECK(cudaMalloc(&bt->start_block, sizeof(int32_t) * cap));
  BT_CHECK(cudaMalloc(&d_out, sizeof(int64_t) * 3));
  if (offsets_bits == 32)
    adj_chain_kernel<int32_t><<<1, 32, 0, st>>>((const int32_t*)d_offsets, N, hdr,
                                                 adj_block_bytes, bt->start_node,
                                                 bt->start_block, cap, d_out);
  else
    adj_chain_kernel<int64_t><<<1, 32, 0, st>>>((const int64_t*)d_offsets, N, hdr,
                                                 adj_block_bytes, bt->start_node,
                                                 bt->start_block, cap, d_out);
  BT_CHECK(cudaGetLastError());
  BT_CHECK(cudaMemcpyAsync(host_out, d_out, sizeof(host_out), cudaMemcpyDeviceToHost, st));
  BT_CHECK(cudaStreamSynchronize(st));
  if (host_out[2]) {
    snprintf(err, errlen, "block table overflow (bound %lld)", (long long)cap);
    rc = cudaErrorInvalidValue;
    goto done;
  }
  bt->n_starts = host_out[0];
  bt->n_blocks = host_out[1];

  BT_CHECK(cudaMalloc(&flags, N));
  BT_CHECK(cudaMalloc(&rank, sizeof(int32_t) * (N + 1)));
  BT_CHECK(cudaMalloc(&scratch, sizeof(int64_t) * scan_scratch_elems(1, N)));
  BT_CHECK(cudaMemsetAsync(scratch, 0, sizeof(int64_t) * scan_scratch_elems(1, N), st));
  tile_flags_kernel<<<grid, 256, 0, st>>>(flags, N, rows_per_feat_block);
  tile_flag_starts_kernel<<<grid, 256, 0, st>>>(flags, bt->start_node, bt->n_starts);
  BT_CHECK(cudaGetLastError());
  BT_CHECK((seg_scan<uint8_t, int32_t>(flags, 0, rank, 0, nullptr, N, 1, N, true, nullptr,
                                       scratch, nullptr, st)));
  BT_CHECK(cudaMemcpyAsync(&T32, rank + N, sizeof(int32_t), cudaMemcpyDeviceToHost, st));
  BT_CHECK(cudaStreamSynchronize(st));
  bt->T = T32;
  BT_CHECK(cudaMalloc(&bt->tile_first, sizeof(int32_t) * (bt->T + 1)));
  BT_CHECK(cudaMalloc(&bt->chunk_tile, sizeof(int32_t) * (C + 1)));
  BT_CHECK(cudaMalloc(&bt->tile_adj_block, sizeof(int32_t) * bt->T));
  BT_CHECK(cudaMalloc(&bt->tile_feat_block, sizeof(int32_t) * bt->T));
  BT_CHECK(cudaMalloc(&bt->fblock_first_tile, sizeof(int32_t) * (bt->n_feat_blocks + 1)));
  BT_CHECK(cudaMalloc(&bt->tile_adj_start, sizeof(int32_t) * bt->T));
  BT_CHECK(cudaMalloc(&bt->run_first_tile, sizeof(int32_t) * (bt->n_starts + 1)));
  BT_CHECK(cudaMalloc(&bt->blk_e0, sizeof(int64_t) * bt->n_blocks));
  BT_CHECK(cudaMalloc(&bt->blk_e1, sizeof(int64_t) * bt->n_blocks));
  tile_compact_kernel<<<grid, 256, 0, st>>>(flags, rank, N, bt->tile_first, bt->chunk_tile);
  tile_blocks_kernel<<<grid, 256, 0, st>>>(bt->tile_first, bt->T, bt->start_node,
                                           bt->start_block, bt->n_starts, rows_per_feat_block,
                                           bt->tile_adj_block, bt->tile_feat_block,
                                           bt->tile_adj_start, bt->run_first_tile);
  if (offsets_bits == 32)
    block_edges_kernel<int32_t><<<grid, 256, 0, st>>>((const int32_t*)d_offsets, N, hdr,
                                                      adj_block_bytes, bt->start_node,
                                                      bt->start_block, bt->n_starts, bt->n_blocks,
                                                      bt->blk_e0, bt->blk_e1);
  else
    block_edges_kernel<int64_t><<<grid, 256, 0, st>>>((const int64_t*)d_offsets, N, hdr,
                                                      adj_block_bytes, bt->start_node,
                                                      bt->start_block, bt->n_starts, bt->n_blocks,
                                                      bt->blk_e0, bt->blk_e1);
  fblock_first_tile_kernel<<<grid, 256, 0, st>>>(bt->tile_first, bt->tile_feat_block, bt->T,
                                                 rows_per_feat_block, bt->n_feat_blocks,
                                                 bt->fblock_first_tile);
  BT_CHECK(cudaGetLastError());
  BT_CHECK(cudaStreamSynchronize(st));

done:
  cudaFree(d_out);
  cudaFree(flags);
  cudaFree(rank);
  cudaFree(scratch);
  if (rc != cudaSuccess) free_block_tables(bt);
  return rc;
}

}  // namespace agnes
