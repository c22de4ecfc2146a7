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
//   - a lane kernel walks all cells, a warp over 32 consecutive cells at a
//     time; a cell of at most 8 entries is resolved by its own thread: its
//     entries become keys (tile-local id << 1 | sampled) in registers,
//     carried with their rows or edge indices through a 19-comparator sorting
//     network, and swept once -- equal ids are adjacent with the frontier
//     entry first, so the first entry of each id is its frontier twin or the
//     new id's first occurrence;
//   - larger cells with samples are queued in cell order (each warp appends
//     its cells in order into its own range; a scan and a copy concatenate
//     the ranges) and resolved one warp per cell on bitmaps over the tile,
//     where every rank is a popcount over per-word prefix counts.
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
  int32_t* q_cells;  // per warp of the lane kernel: its queued cells, at its range's start
  int32_t* q_cnt;    // per warp: how many
  int32_t* q_off;    // exclusive scan of q_cnt (nw + 1)
  int32_t* q_dense;  // the queue, in cell order
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

template <int I, int J>
__device__ __forceinline__ void cmp_swap(int32_t (&k)[kLaneMax], int32_t (&p)[kLaneMax]) {
  const bool sw = k[I] > k[J];
  const int32_t ki = k[I], pi = p[I];
  k[I] = sw ? k[J] : ki;
  p[I] = sw ? p[J] : pi;
  k[J] = sw ? ki : k[J];
  p[J] = sw ? pi : p[J];
}

// Sorts 8 (key, payload) pairs by key in registers: a 19-comparator network
// in six layers.
__device__ __forceinline__ void sort8(int32_t (&k)[kLaneMax], int32_t (&p)[kLaneMax]) {
  cmp_swap<0, 2>(k, p); cmp_swap<1, 3>(k, p); cmp_swap<4, 6>(k, p); cmp_swap<5, 7>(k, p);
  cmp_swap<0, 4>(k, p); cmp_swap<1, 5>(k, p); cmp_swap<2, 6>(k, p); cmp_swap<3, 7>(k, p);
  cmp_swap<0, 1>(k, p); cmp_swap<2, 3>(k, p); cmp_swap<4, 5>(k, p); cmp_swap<6, 7>(k, p);
  cmp_swap<2, 4>(k, p); cmp_swap<3, 5>(k, p);
  cmp_swap<1, 4>(k, p); cmp_swap<3, 6>(k, p);
  cmp_swap<1, 2>(k, p); cmp_swap<3, 4>(k, p); cmp_swap<5, 6>(k, p);
}

// Resolves one cell with samples and at most kLaneMax entries in one thread.
template <bool kPacked>
__device__ __forceinline__ void thread_cell(const CellsArgs& a, int64_t cell, const CellFacts& c) {
  const int32_t n = c.fn + c.sn;
  const int32_t tb = __ldg(a.tile_first + c.t);
  int32_t key[kLaneMax], pay[kLaneMax];
#pragma unroll
  for (int q = 0; q < kLaneMax; ++q) {
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
  sort8(key, pay);
  // sweep: the first entry of each id is its frontier twin (sorted first) or,
  // without one, the new id's first occurrence
  const int64_t jrow = (int64_t)c.j * a.capK;
  int32_t* col = a.col + (int64_t)c.j * a.ecap;
  int2* tmp = a.tmp + c.fo + c.so;
  int32_t prev = -1, cnt_new = 0, cnt_keep = 0, cur = 0;  // cur: col of the current id
#pragma unroll
  for (int q = 0; q < kLaneMax; ++q) {
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

// Walks every cell, a warp over 32 consecutive cells at a time; each warp
// takes a contiguous range of batches and appends its queued cells (with
// samples and more than kLaneMax entries) in order at the start of its own
// range of q_cells (q_cnt[warp] of them).
template <bool kPacked>
__global__ void __launch_bounds__(kThreads, 6) dedup_lane_kernel(CellsArgs a) {
  grid_dep_wait();
  if (failed(a.status)) return;
  const int lane = lane_id();
  const int64_t nbatch = (a.ncells + 31) >> 5;
  const int64_t gw = blockIdx.x * (int64_t)kWarps + (threadIdx.x >> 5);
  const int64_t nw = (int64_t)gridDim.x * kWarps;
  const int64_t b_lo = gw * nbatch / nw, b_hi = (gw + 1) * nbatch / nw;
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
    if (has && c.sn > 0 && n <= kLaneMax) thread_cell<kPacked>(a, cell, c);
  }
  if (lane == 0) a.q_cnt[gw] = queued;
}

// The queue in cell order: q_off = the exclusive scan of the warps' counts
// (one CTA) ...
__global__ void __launch_bounds__(1024) queue_offsets_kernel(const int32_t* q_cnt, int32_t nw,
                                                             int32_t* q_off,
                                                             const int32_t* status) {
  grid_dep_wait();
  if (failed(status)) return;
  __shared__ int32_t wsum[32];
  __shared__ int32_t carry;
  if (threadIdx.x == 0) carry = 0;
  __syncthreads();
  const int lane = lane_id(), w = threadIdx.x >> 5;
  for (int32_t base = 0; base < nw; base += 1024) {
    const int32_t i = base + threadIdx.x;
    const int32_t v = i < nw ? q_cnt[i] : 0;
    const int32_t incl = warp_incl_scan(v);
    if (lane == 31) wsum[w] = incl;
    __syncthreads();
    if (w == 0) {
      const int32_t t = wsum[lane];
      wsum[lane] = warp_incl_scan(t) - t;
    }
    __syncthreads();
    if (i < nw) q_off[i] = carry + wsum[w] + incl - v;
    __syncthreads();
    if (threadIdx.x == 1023) carry += wsum[31] + incl;
    __syncthreads();
  }
  if (threadIdx.x == 0) q_off[nw] = carry;
}

// ... then each warp's run copied to q_dense[q_off[warp] ...).
__global__ void __launch_bounds__(kThreads) queue_compact_kernel(CellsArgs a, int32_t nw) {
  grid_dep_wait();
  if (failed(a.status)) return;
  const int lane = lane_id();
  const int64_t nbatch = (a.ncells + 31) >> 5;
  const int64_t nwarps = (int64_t)gridDim.x * kWarps;
  for (int64_t r = blockIdx.x * (int64_t)kWarps + (threadIdx.x >> 5); r < nw; r += nwarps) {
    const int64_t src = (r * nbatch / nw) << 5;
    const int32_t dst = a.q_off[r], cnt = a.q_off[r + 1] - dst;
    for (int32_t i = lane; i < cnt; i += 32) a.q_dense[dst + i] = a.q_cells[src + i];
  }
}

// ---- queued cells: a warp each, on bitmaps over the tile --------------------------

// A warp's shared-memory scratch: kTileWords (128) words each, lane l owning
// words 4l .. 4l+3, which it reads and writes as one 16-byte vector
// (conflict-free).
struct TileScratch {
  uint32_t* D;  // frontier ids
  uint32_t* S;  // sampled ids, then N = S & ~D, the new ids
  uint32_t* C;  // new ids already entered in the next frontier cell
  int32_t* pD;  // frontier ids below word w
  int32_t* pN;  // new ids below word w
};

template <bool kPacked>
__global__ void __launch_bounds__(kThreads, 8) dedup_tile_kernel(CellsArgs a, int32_t nw) {
  grid_dep_wait();
  if (failed(a.status)) return;
  __shared__ __align__(16) uint32_t D_s[kWarps][kTileWords];
  __shared__ __align__(16) uint32_t S_s[kWarps][kTileWords];
  __shared__ __align__(16) uint32_t C_s[kWarps][kTileWords];
  __shared__ __align__(16) int32_t pD_s[kWarps][kTileWords];
  __shared__ __align__(16) int32_t pN_s[kWarps][kTileWords];
  const int warp = threadIdx.x >> 5, lane = lane_id();
  const TileScratch t{D_s[warp], S_s[warp], C_s[warp], pD_s[warp], pN_s[warp]};
  const int32_t total = a.q_off[nw];
  const int64_t nwarps = (int64_t)gridDim.x * kWarps;
  for (int64_t q = blockIdx.x * (int64_t)kWarps + warp; q < total; q += nwarps) {
    const int64_t cell = a.q_dense[q];
    const CellFacts c = cell_facts(a, cell);
    const int32_t base = __ldg(a.tile_first + c.t);
    // mark D and S
    const uint4 z = make_uint4(0u, 0u, 0u, 0u);
    reinterpret_cast<uint4*>(t.D)[lane] = z;
    reinterpret_cast<uint4*>(t.S)[lane] = z;
    reinterpret_cast<uint4*>(t.C)[lane] = z;
    __syncwarp();
    for (int32_t i0 = lane; i0 < c.fn; i0 += 128) {  // four entries in flight per lane
      int32_t v[4];
#pragma unroll
      for (int k = 0; k < 4; ++k)
        v[k] = i0 + 32 * k < c.fn ? a.fb_id[c.fo + i0 + 32 * k] - base : -1;
#pragma unroll
      for (int k = 0; k < 4; ++k)
        if (v[k] >= 0) atomicOr(t.D + (v[k] >> 5), 1u << (v[k] & 31));
    }
    for (int32_t i0 = lane; i0 < c.sn; i0 += 128) {
      int32_t v[4];
#pragma unroll
      for (int k = 0; k < 4; ++k)
        v[k] = i0 + 32 * k < c.sn ? sampled_entry<kPacked>(a, c.so + i0 + 32 * k, base).x : -1;
#pragma unroll
      for (int k = 0; k < 4; ++k)
        if (v[k] >= 0) atomicOr(t.S + (v[k] >> 5), 1u << (v[k] & 31));
    }
    __syncwarp();
    // N = S & ~D and the per-word prefix counts of D and N
    const uint4 d = reinterpret_cast<const uint4*>(t.D)[lane];
    const uint4 sv = reinterpret_cast<const uint4*>(t.S)[lane];
    const uint4 nv = make_uint4(sv.x & ~d.x, sv.y & ~d.y, sv.z & ~d.z, sv.w & ~d.w);
    const int32_t cd0 = __popc(d.x), cd1 = __popc(d.y), cd2 = __popc(d.z), cd3 = __popc(d.w);
    const int32_t cn0 = __popc(nv.x), cn1 = __popc(nv.y), cn2 = __popc(nv.z), cn3 = __popc(nv.w);
    const int32_t lane_d = cd0 + cd1 + cd2 + cd3, lane_n = cn0 + cn1 + cn2 + cn3;
    const int32_t ed = warp_incl_scan(lane_d) - lane_d;
    const int32_t en_incl = warp_incl_scan(lane_n);
    const int32_t en = en_incl - lane_n;
    reinterpret_cast<int4*>(t.pD)[lane] =
        make_int4(ed, ed + cd0, ed + cd0 + cd1, ed + cd0 + cd1 + cd2);
    reinterpret_cast<int4*>(t.pN)[lane] =
        make_int4(en, en + cn0, en + cn0 + cn1, en + cn0 + cn1 + cn2);
    reinterpret_cast<uint4*>(t.S)[lane] = nv;
    if (lane == 31) {
      a.newcnt[cell] = en_incl;
      a.nfcnt[cell] = c.fn + en_incl;
    }
    __syncwarp();
    const uint32_t* N = t.S;
    const int64_t jrow = (int64_t)c.j * a.capK;
    int2* tmp = a.tmp + c.fo + c.so;
    // frontier entries (sorted: entry i has i frontier ids below it) keep
    // their rows; below them in the next cell also lie the new ids below
    for (int32_t i = lane; i < c.fn; i += 32) {
      const int32_t v = a.fb_id[c.fo + i] - base;
      const int32_t w = v >> 5;
      const uint32_t below = (1u << (v & 31)) - 1u;
      tmp[i + t.pN[w] + __popc(N[w] & below)] = make_int2(base + v, a.fb_pos[c.fo + i]);
    }
    int32_t* col = a.col + (int64_t)c.j * a.ecap;
    for (int32_t i = lane; i < c.sn; i += 32) {
      const int2 e = sampled_entry<kPacked>(a, c.so + i, base);
      const int32_t v = e.x;
      const int32_t w = v >> 5;
      const uint32_t bit = 1u << (v & 31), below = bit - 1u;
      const uint32_t dw = t.D[w];
      const int32_t rd = t.pD[w] + __popc(dw & below);  // frontier ids below
      if (dw & bit) {
        col[e.y] = (int32_t)(a.fb_pos[c.fo + rd] - jrow);
      } else {
        const int32_t rn = t.pN[w] + __popc(N[w] & below);  // new ids below
        col[e.y] = -1 - rn;
        if ((atomicOr(t.C + w, bit) & bit) == 0u)  // the id's first entry enters the cell
          tmp[rd + rn] = make_int2(base + v, -1 - rn);
      }
    }
    __syncwarp();  // the scratch is rewritten by the next cell
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
  a.status = h.status;
  return a;
}

template <bool kPacked>
cudaError_t launch_cells(const CellsArgs& a, int32_t q_warps_cap, int num_sms, cudaStream_t st) {
  const int grid = resident_grid((const void*)dedup_lane_kernel<kPacked>, kThreads, num_sms);
  const int nw = grid * kWarps;
  if (nw > q_warps_cap) return cudaErrorInvalidValue;
  dedup_lane_kernel<kPacked><<<grid, kThreads, 0, st>>>(a);
  queue_offsets_kernel<<<1, 1024, 0, st>>>(a.q_cnt, nw, a.q_off, a.status);
  queue_compact_kernel<<<resident_grid((const void*)queue_compact_kernel, kThreads, num_sms),
                         kThreads, 0, st>>>(a, nw);
  dedup_tile_kernel<kPacked><<<resident_grid((const void*)dedup_tile_kernel<kPacked>, kThreads,
                                             num_sms),
                               kThreads, 0, st>>>(a, nw);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_dedup_cells(const HopArgs& h, const DedupBufs& d, int num_sms,
                               cudaStream_t st) {
  const CellsArgs a = cells_args(h, d);
  return h.sb_packed ? launch_cells<true>(a, d.q_warps_cap, num_sms, st)
                     : launch_cells<false>(a, d.q_warps_cap, num_sms, st);
}

}  // namespace agnes
