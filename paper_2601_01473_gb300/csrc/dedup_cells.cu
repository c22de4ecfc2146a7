// dedup_cells.cu -- the default frontier's resolution of one hop's cells
// (Algorithm 1: N^j_out <- N^j_out u Sample(j, ...); src_h = dst_h ++ new_h,
// dst_{h+1} = src_h).  A cell (t, j) of the bucket matrix holds D, minibatch
// j's frontier ids in tile t (ascending), and S, its sampled ids there.
// Resolving it gives, with ranks local to the cell:
//   newcnt / nfcnt   |S \ D| and |D u (S \ D)|;
//   col[e]           the frontier twin's index in dst_h, or -(1 + r) for the
//                    r-th smallest new id of the cell;
//   tmp              the next frontier cell D u new in ascending id, a new id
//                    with x = -(1 + r), a frontier id with its row;
// dedup.cu's scans, col fix-up and compaction then turn the local ranks into
// final indices (coalesced passes over edges and over the next bucket).
//
// Work layout.  Cells are small on average, but the entries concentrate in
// the larger cells of the tiles that hold the graph's hubs (at rmat100m's hop
// 3, cells of more than 32 entries hold over half of them), so:
//   - a lane kernel walks all cells in chunks of 256 taken from a counter, a
//     warp over 32 consecutive cells at a time; a cell of at most 8 entries
//     is resolved by its own thread: its entries become keys (tile-local id
//     << 1 | sampled) in registers, carried with their rows or edge indices
//     through a 5- or 19-comparator sorting network, and swept once -- equal
//     ids are adjacent with the frontier entry first, so the first entry of
//     each id is its frontier twin or the new id's first occurrence;
//   - larger cells with samples are queued in cell order (each chunk's cells
//     in order at the start of its own range; a scan and a copy concatenate
//     the ranges) and resolved one warp per cell on bitmaps over the tile,
//     where every rank is a popcount over per-word prefix counts.
// The sampled bucket is either (id, edge index) pairs or, when the hop's
// edge indices fit 20 bits, packed words edge index << 12 | tile-local id
// (the kernels' kPacked).
#include "common.cuh"
#include "internal.h"

namespace agnes {

namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kLaneMax = kDedupLaneMax;  // entries a single thread resolves
constexpr unsigned kFull = 0xffffffffu;
constexpr int32_t kNoKey = 0x7fffffff;

static_assert(kLaneMax == 8, "the 19-comparator network is for 8 keys");
static_assert(kTileWords == 128, "a lane owns four words of the tile bitmap");

struct CellsArgs {
  int64_t ncells;
  int32_t H;
  int64_t capK, ecap;
  const int32_t* tile_first;
  const int32_t* fb_id;  // frontier bucket: ids ascending inside a cell
  const int32_t* fb_pos;
  const int32_t* fcell_off;
  const int2* sb;  // sampled bucket: (id, edge index in the minibatch), or packed 4-byte
                   // entries edge index << 12 | tile-local id (the kernels' kPacked)
  const int32_t* soff;
  const int32_t* tile_adj_block;
  uint8_t* adj_flags;
  int32_t* newcnt;
  int32_t* nfcnt;
  int2* tmp;     // per cell at fcell_off + soff: next-frontier entries, local ranks
  int32_t* col;  // H x ecap
  int32_t* q_cells;  // per chunk of kChunkCells cells: its queued cells, at the chunk's start
  int32_t* q_cnt;    // per chunk: how many
  int32_t* q_off;    // exclusive scan of q_cnt (nchunks + 1)
  int32_t* q_dense;  // the queue, in cell order
  int32_t* q_next;   // the lane kernel's next chunk (zero between launches)
  const int32_t* status;
};

struct CellFacts {
  int32_t fo, fn, so, sn, t, j;
};

// Cell (t, j) = t * H + j.
__device__ __forceinline__ CellFacts cell_facts(const CellsArgs& a, int64_t cell, int32_t t,
                                                int32_t j) {
  CellFacts c;
  c.fo = a.fcell_off[cell];
  c.fn = a.fcell_off[cell + 1] - c.fo;
  c.so = a.soff[cell];
  c.sn = a.soff[cell + 1] - c.so;
  c.t = t;
  c.j = j;
  return c;
}

__device__ __forceinline__ CellFacts cell_facts(const CellsArgs& a, int64_t cell) {
  const int32_t t = (int32_t)((uint32_t)cell / (uint32_t)a.H);  // cells < 2^31
  return cell_facts(a, cell, t, (int32_t)cell - t * a.H);
}

// Sampled entry i of the bucket as (tile-local id, edge index); base is the
// tile's first id.
template <bool kPacked>
__device__ __forceinline__ int2 sampled_entry(const CellsArgs& a, int32_t i, int32_t base) {
  if constexpr (kPacked) {
    const uint32_t v = reinterpret_cast<const uint32_t*>(a.sb)[i];
    return make_int2((int32_t)(v & 0xfffu), (int32_t)(v >> 12));
  } else {
    const int2 e = a.sb[i];
    return make_int2(e.x - base, e.y);
  }
}

// ---- cells of at most kLaneMax entries: a thread each ---------------------------

template <int I, int J, int W>
__device__ __forceinline__ void cmp_swap(int32_t (&k)[W], int32_t (&p)[W]) {
  const bool sw = k[I] > k[J];
  const int32_t ki = k[I], pi = p[I];
  k[I] = sw ? k[J] : ki;
  p[I] = sw ? p[J] : pi;
  k[J] = sw ? ki : k[J];
  p[J] = sw ? pi : p[J];
}

// Sorts 4 (key, payload) pairs by key in registers: 5 comparators.
__device__ __forceinline__ void sort_net(int32_t (&k)[4], int32_t (&p)[4]) {
  cmp_swap<0, 1>(k, p); cmp_swap<2, 3>(k, p);
  cmp_swap<0, 2>(k, p); cmp_swap<1, 3>(k, p);
  cmp_swap<1, 2>(k, p);
}

// Sorts 8 (key, payload) pairs by key in registers: a 19-comparator network
// in six layers.
__device__ __forceinline__ void sort_net(int32_t (&k)[8], int32_t (&p)[8]) {
  cmp_swap<0, 2>(k, p); cmp_swap<1, 3>(k, p); cmp_swap<4, 6>(k, p); cmp_swap<5, 7>(k, p);
  cmp_swap<0, 4>(k, p); cmp_swap<1, 5>(k, p); cmp_swap<2, 6>(k, p); cmp_swap<3, 7>(k, p);
  cmp_swap<0, 1>(k, p); cmp_swap<2, 3>(k, p); cmp_swap<4, 5>(k, p); cmp_swap<6, 7>(k, p);
  cmp_swap<2, 4>(k, p); cmp_swap<3, 5>(k, p);
  cmp_swap<1, 4>(k, p); cmp_swap<3, 6>(k, p);
  cmp_swap<1, 2>(k, p); cmp_swap<3, 4>(k, p); cmp_swap<5, 6>(k, p);
}

// Resolves one cell with samples and at most W (4 or 8, kLaneMax at most)
// entries in one thread.
template <bool kPacked, int W>
__device__ __forceinline__ void thread_cell(const CellsArgs& a, int64_t cell, const CellFacts& c) {
  const int32_t n = c.fn + c.sn;
  const int32_t tb = __ldg(a.tile_first + c.t);
  int32_t key[W], pay[W];
#pragma unroll
  for (int q = 0; q < W; ++q) {
    key[q] = kNoKey;
    pay[q] = 0;
    if (q < c.fn) {
      key[q] = (a.fb_id[c.fo + q] - tb) << 1;
      pay[q] = a.fb_pos[c.fo + q];
    } else if (q < n) {
      const int2 e = sampled_entry<kPacked>(a, c.so + (q - c.fn), tb);
      key[q] = (e.x << 1) | 1;
      pay[q] = e.y;
    }
  }
  sort_net(key, pay);
  // sweep: the first entry of each id is its frontier twin (sorted first) or,
  // without one, the new id's first occurrence
  const int64_t jrow = (int64_t)c.j * a.capK;
  int32_t* col = a.col + (int64_t)c.j * a.ecap;
  int2* tmp = a.tmp + c.fo + c.so;
  int32_t prev = -1, cnt_new = 0, cnt_keep = 0, cur = 0;  // cur: col of the current id
#pragma unroll
  for (int q = 0; q < W; ++q) {
    if (key[q] != kNoKey) {
      const int32_t lu = key[q] >> 1;
      const bool sampled = key[q] & 1;
      if (lu != prev) {  // the id's first entry: it enters the next frontier cell
        int32_t x;
        if (!sampled) {
          x = pay[q];
          cur = (int32_t)(x - jrow);
        } else {
          x = -1 - cnt_new;
          cur = x;
          ++cnt_new;
        }
        tmp[cnt_keep++] = make_int2(tb + lu, x);
      }
      if (sampled) col[pay[q]] = cur;
      prev = lu;
    }
  }
  a.newcnt[cell] = cnt_new;
  a.nfcnt[cell] = c.fn + cnt_new;
}

// Walks every cell, a warp over 32 consecutive cells at a time.  Warps take
// chunks of kChunkCells cells from a counter (cells differ widely in cost, so
// fixed ranges would leave warps idle); each appends its queued cells (with
// samples and more than kLaneMax entries) in order at the start of the
// chunk's range of q_cells (q_cnt[chunk] of them).
constexpr int kChunkCells = kDedupChunkCells;
constexpr int kChunkBatches = kChunkCells / 32;

// Batches [b_lo, b_hi) of one chunk.
template <bool kPacked>
__device__ __forceinline__ void lane_chunk(const CellsArgs& a, int lane, int64_t b_lo,
                                           int64_t b_hi, int32_t chunk) {
  int32_t queued = 0;
  // the lane's cell (t, j), advanced by 32 cells per batch
  int32_t t = (int32_t)((uint32_t)((b_lo << 5) + lane) / (uint32_t)a.H);  // cells < 2^31
  int32_t j = (int32_t)((b_lo << 5) + lane) - t * a.H;
  for (int64_t b = b_lo; b < b_hi; ++b) {
    const int64_t cell = (b << 5) + lane;
    const bool has = cell < a.ncells;
    CellFacts c{0, 0, 0, 0, 0, 0};
    if (has) c = cell_facts(a, cell, t, j);
    for (j += 32; j >= a.H; j -= a.H) ++t;
    const int32_t n = c.fn + c.sn;
    if (has && c.fn > 0) a.adj_flags[a.tile_adj_block[c.t]] = 1;
    if (has && c.sn == 0) {  // nothing sampled: the compaction copies the frontier cell
      a.newcnt[cell] = 0;
      a.nfcnt[cell] = c.fn;
    }
    const unsigned qm = __ballot_sync(kFull, has && c.sn > 0 && n > kLaneMax);
    if ((qm >> lane) & 1u)
      a.q_cells[(b_lo << 5) + queued + __popc(qm & ((1u << lane) - 1u))] = (int32_t)cell;
    queued += __popc(qm);
    // the warp takes the 4-entry network unless one of its cells needs 8
    const bool mine = has && c.sn > 0 && n <= kLaneMax;
    if (__any_sync(kFull, mine && n > 4)) {
      if (mine) thread_cell<kPacked, 8>(a, cell, c);
    } else if (mine) {
      thread_cell<kPacked, 4>(a, cell, c);
    }
  }
  if (lane == 0) a.q_cnt[chunk] = queued;
}

template <bool kPacked>
__global__ void __launch_bounds__(kThreads, 6) dedup_lane_kernel(CellsArgs a) {
  grid_dep_wait();
  if (failed(a.status)) return;
  const int lane = lane_id();
  const int64_t nbatch = (a.ncells + 31) >> 5;
  const int32_t nchunks = (int32_t)((a.ncells + kChunkCells - 1) / kChunkCells);
  for (;;) {
    int32_t chunk = 0;
    if (lane == 0) chunk = atomicAdd(a.q_next, 1);
    chunk = __shfl_sync(kFull, chunk, 0);
    if (chunk >= nchunks) break;
    lane_chunk<kPacked>(a, lane, (int64_t)chunk * kChunkBatches,
                        min((int64_t)(chunk + 1) * kChunkBatches, nbatch), chunk);
  }
}

// The queue in cell order: q_off = the exclusive scan of the chunks' counts
// (one CTA, four counts per thread and round; it also rewinds the lane
// kernel's chunk counter) ...
__global__ void __launch_bounds__(1024) queue_offsets_kernel(const int32_t* q_cnt, int32_t nw,
                                                             int32_t* q_off, int32_t* q_next,
                                                             const int32_t* status) {
  grid_dep_wait();
  if (threadIdx.x == 0) *q_next = 0;
  if (failed(status)) return;
  __shared__ int32_t wsum[32];
  __shared__ int32_t carry;
  if (threadIdx.x == 0) carry = 0;
  __syncthreads();
  const int lane = lane_id(), w = threadIdx.x >> 5;
  for (int32_t base = 0; base < nw; base += 4096) {
    const int32_t i = base + 4 * (int32_t)threadIdx.x;
    int32_t v[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) v[k] = i + k < nw ? q_cnt[i + k] : 0;
    const int32_t mine = v[0] + v[1] + v[2] + v[3];
    const int32_t incl = warp_incl_scan(mine);
    if (lane == 31) wsum[w] = incl;
    __syncthreads();
    if (w == 0) {
      const int32_t t = wsum[lane];
      wsum[lane] = warp_incl_scan(t) - t;
    }
    __syncthreads();
    int32_t run = carry + wsum[w] + incl - mine;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      if (i + k < nw) q_off[i + k] = run;
      run += v[k];
    }
    __syncthreads();
    if (threadIdx.x == 1023) carry = run;
    __syncthreads();
  }
  if (threadIdx.x == 0) q_off[nw] = carry;
}

// ... then each chunk's run copied to q_dense[q_off[chunk] ...).
__global__ void __launch_bounds__(kThreads) queue_compact_kernel(CellsArgs a, int32_t nw) {
  grid_dep_wait();
  if (failed(a.status)) return;
  const int lane = lane_id();
  const int64_t nwarps = (int64_t)gridDim.x * kWarps;
  for (int64_t r = blockIdx.x * (int64_t)kWarps + (threadIdx.x >> 5); r < nw; r += nwarps) {
    const int64_t src = r * kChunkCells;
    const int32_t dst = a.q_off[r], cnt = a.q_off[r + 1] - dst;
    for (int32_t i = lane; i < cnt; i += 32) a.q_dense[dst + i] = a.q_cells[src + i];
  }
}

// ---- queued cells: a warp each, on bitmaps over the tile --------------------------

// Marks entries 0 .. n-1 of a cell in a bitmap: put(get(i)) per entry, the
// lanes taking entries lane, lane + 32, ...; past 64 entries four loads per
// lane are issued before their marks.
template <typename Get, typename Put>
__device__ __forceinline__ void mark_entries(int32_t n, int lane, Get get, Put put) {
  if (n <= 64) {
    for (int32_t i = lane; i < n; i += 32) put(get(i));
    return;
  }
  for (int32_t i0 = lane; i0 < n; i0 += 128) {
    int32_t v[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) v[k] = i0 + 32 * k < n ? get(i0 + 32 * k) : -1;
#pragma unroll
    for (int k = 0; k < 4; ++k)
      if (v[k] >= 0) put(v[k]);
  }
}

// A warp's shared-memory scratch, lane l owning words 4l .. 4l+3 of each
// bitmap over the tile (kTileWords = 128 words), read and written as one
// 16-byte vector (conflict-free):
//   D[w]   frontier ids of word w;
//   N[w]   sampled ids, then the new ids S & ~D once both are marked;
//   P[w]   frontier ids below word w << 16 | new ids below word w (each at
//          most 4096, so the two halves add without carries);
//   C[w]   new ids already entered in the next frontier cell.
struct TileResolver {
  const uint32_t* D;
  const uint32_t* N;
  const uint32_t* P;
  uint32_t* C;
  int2* tmp;            // the cell's next-frontier entries
  int32_t* col;         // the minibatch's col
  const int32_t* fpos;  // the cell's frontier rows
  int32_t base, jrow;

  // Frontier entry i (sorted: i frontier ids lie below it) with tile-local id
  // v keeps its row; below it in the next cell also lie the new ids below v.
  __device__ __forceinline__ void frontier(int32_t i, int32_t v, int32_t row) const {
    const int32_t w = v >> 5;
    const uint32_t below = (1u << (v & 31)) - 1u;
    tmp[i + (int32_t)(P[w] & 0xffffu) + __popc(N[w] & below)] = make_int2(base + v, row);
  }

  // Sampled entry (tile-local id, edge index): col is its frontier twin's
  // row in dst, or -(1 + r) for the r-th new id of the cell, whose first
  // entry enters the next frontier cell.
  __device__ __forceinline__ void sampled(int2 e) const {
    const int32_t v = e.x;
    const int32_t w = v >> 5;
    const uint32_t bit = 1u << (v & 31), below = bit - 1u;
    const uint32_t dw = D[w];
    const uint32_t pw = P[w];
    const int32_t rd = (int32_t)(pw >> 16) + __popc(dw & below);  // frontier ids below
    if (dw & bit) {
      col[e.y] = fpos[rd] - jrow;
    } else {
      const int32_t rn = (int32_t)(pw & 0xffffu) + __popc(N[w] & below);  // new ids below
      col[e.y] = -1 - rn;
      if ((atomicOr(C + w, bit) & bit) == 0u) tmp[rd + rn] = make_int2(base + v, -1 - rn);
    }
  }
};

// One warp per queued cell.  A cell of at most 32 frontier and 64 sampled
// entries (most queued cells) is read once into registers, with all its loads
// in flight together, and resolved from there; larger cells are walked twice
// (mark, resolve).  Each warp loads the next queued cell's offsets while it
// resolves the current one.
template <bool kPacked>
__global__ void __launch_bounds__(kThreads, 5) dedup_tile_kernel(CellsArgs a, int32_t nw) {
  grid_dep_wait();
  if (failed(a.status)) return;
  __shared__ __align__(16) uint32_t D_s[kWarps][kTileWords];
  __shared__ __align__(16) uint32_t N_s[kWarps][kTileWords];
  __shared__ __align__(16) uint32_t P_s[kWarps][kTileWords];
  __shared__ __align__(16) uint32_t C_s[kWarps][kTileWords];
  const int warp = threadIdx.x >> 5, lane = lane_id();
  uint32_t* D = D_s[warp];
  uint32_t* N = N_s[warp];
  uint32_t* P = P_s[warp];
  uint32_t* C = C_s[warp];
  const int32_t total = a.q_off[nw];
  const int32_t nwarps = (int32_t)gridDim.x * kWarps;
  int32_t q = (int32_t)blockIdx.x * kWarps + warp;
  int32_t cell = q < total ? a.q_dense[q] : 0;
  CellFacts c = cell_facts(a, cell);
  for (; q < total; q += nwarps) {
    const int32_t next = q + nwarps < total ? a.q_dense[q + nwarps] : cell;
    const CellFacts cn = cell_facts(a, next);
    const int32_t base = __ldg(a.tile_first + c.t);
    const int32_t* fid = a.fb_id + c.fo;
    const int32_t* fpos = a.fb_pos + c.fo;
    const bool small = c.fn <= 32 && c.sn <= 64;  // warp-uniform
    int32_t fv = -1, fr = 0;
    int2 s0 = make_int2(-1, 0), s1 = make_int2(-1, 0);
    if (small) {
      if (lane < c.fn) {
        fv = fid[lane] - base;
        fr = fpos[lane];
      }
      if (lane < c.sn) s0 = sampled_entry<kPacked>(a, c.so + lane, base);
      if (lane + 32 < c.sn) s1 = sampled_entry<kPacked>(a, c.so + lane + 32, base);
    }
    // mark D and S
    const uint4 z = make_uint4(0u, 0u, 0u, 0u);
    reinterpret_cast<uint4*>(D)[lane] = z;
    reinterpret_cast<uint4*>(N)[lane] = z;
    reinterpret_cast<uint4*>(C)[lane] = z;
    __syncwarp();
    if (small) {
      if (fv >= 0) atomicOr(D + (fv >> 5), 1u << (fv & 31));
      if (s0.x >= 0) atomicOr(N + (s0.x >> 5), 1u << (s0.x & 31));
      if (s1.x >= 0) atomicOr(N + (s1.x >> 5), 1u << (s1.x & 31));
    } else {
      mark_entries(
          c.fn, lane, [&](int32_t i) { return fid[i] - base; },
          [&](int32_t v) { atomicOr(D + (v >> 5), 1u << (v & 31)); });
      mark_entries(
          c.sn, lane, [&](int32_t i) { return sampled_entry<kPacked>(a, c.so + i, base).x; },
          [&](int32_t v) { atomicOr(N + (v >> 5), 1u << (v & 31)); });
    }
    __syncwarp();
    // N = S & ~D and the per-word prefix counts, both halves in one scan
    const uint4 d = reinterpret_cast<const uint4*>(D)[lane];
    uint4 nv = reinterpret_cast<const uint4*>(N)[lane];
    nv.x &= ~d.x;
    nv.y &= ~d.y;
    nv.z &= ~d.z;
    nv.w &= ~d.w;
    const uint32_t k0 = ((uint32_t)__popc(d.x) << 16) | (uint32_t)__popc(nv.x);
    const uint32_t k1 = ((uint32_t)__popc(d.y) << 16) | (uint32_t)__popc(nv.y);
    const uint32_t k2 = ((uint32_t)__popc(d.z) << 16) | (uint32_t)__popc(nv.z);
    const uint32_t k3 = ((uint32_t)__popc(d.w) << 16) | (uint32_t)__popc(nv.w);
    const uint32_t mine = k0 + k1 + k2 + k3;
    const uint32_t incl = warp_incl_scan(mine);
    const uint32_t ex = incl - mine;
    reinterpret_cast<uint4*>(P)[lane] = make_uint4(ex, ex + k0, ex + k0 + k1, ex + k0 + k1 + k2);
    reinterpret_cast<uint4*>(N)[lane] = nv;
    if (lane == 31) {
      a.newcnt[cell] = (int32_t)(incl & 0xffffu);
      a.nfcnt[cell] = c.fn + (int32_t)(incl & 0xffffu);
    }
    __syncwarp();
    const TileResolver r{D, N, P, C, a.tmp + c.fo + c.so, a.col + (int64_t)c.j * a.ecap, fpos,
                         base, (int32_t)((int64_t)c.j * a.capK)};
    if (small) {
      if (fv >= 0) r.frontier(lane, fv, fr);
      if (s0.x >= 0) r.sampled(s0);
      if (s1.x >= 0) r.sampled(s1);
    } else {
      for (int32_t i = lane; i < c.fn; i += 32) r.frontier(i, fid[i] - base, fpos[i]);
      for (int32_t i = lane; i < c.sn; i += 32) r.sampled(sampled_entry<kPacked>(a, c.so + i, base));
    }
    __syncwarp();  // the scratch is rewritten by the next cell
    cell = next;
    c = cn;
  }
}

CellsArgs cells_args(const HopArgs& h, const DedupBufs& d) {
  CellsArgs a;
  a.ncells = (int64_t)h.T * h.H;
  a.H = h.H;
  a.capK = h.capK;
  a.ecap = h.ecap;
  a.tile_first = h.tile_first;
  a.fb_id = d.fb_id;
  a.fb_pos = d.fb_pos;
  a.fcell_off = d.fcell_off;
  a.sb = d.sb;
  a.soff = d.soff;
  a.tile_adj_block = d.tile_adj_block;
  a.adj_flags = d.adj_flags;
  a.newcnt = d.newcnt;
  a.nfcnt = d.nfcnt;
  a.tmp = d.tmp;
  a.col = d.col;
  a.q_cells = d.q_cells;
  a.q_cnt = d.q_cnt;
  a.q_off = d.q_off;
  a.q_dense = d.q_dense;
  a.q_next = d.q_next;
  a.status = h.status;
  return a;
}

template <bool kPacked>
cudaError_t launch_cells(const CellsArgs& a, int32_t q_chunks_cap, int num_sms, cudaStream_t st) {
  const int grid = resident_grid((const void*)dedup_lane_kernel<kPacked>, kThreads, num_sms);
  const int64_t nw = (a.ncells + kChunkCells - 1) / kChunkCells;  // chunks
  if (nw > q_chunks_cap) return cudaErrorInvalidValue;
  dedup_lane_kernel<kPacked><<<grid, kThreads, 0, st>>>(a);
  queue_offsets_kernel<<<1, 1024, 0, st>>>(a.q_cnt, (int32_t)nw, a.q_off, a.q_next, a.status);
  queue_compact_kernel<<<resident_grid((const void*)queue_compact_kernel, kThreads, num_sms),
                         kThreads, 0, st>>>(a, (int32_t)nw);
  dedup_tile_kernel<kPacked><<<resident_grid((const void*)dedup_tile_kernel<kPacked>, kThreads,
                                             num_sms),
                               kThreads, 0, st>>>(a, (int32_t)nw);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_dedup_cells(const HopArgs& h, const DedupBufs& d, int num_sms,
                               cudaStream_t st) {
  const CellsArgs a = cells_args(h, d);
  return h.sb_packed ? launch_cells<true>(a, d.q_chunks_cap, num_sms, st)
                     : launch_cells<false>(a, d.q_chunks_cap, num_sms, st);
}

}  // namespace agnes
