// dedup.cu -- per-minibatch union / dedup and relabelling of a hop's samples
// (Algorithm 1: N^j_out <- N^j_out u Sample(j, ...), N_in <- N_out).
//
// The sampled ids of every minibatch are bucketed by (tile, minibatch) cell
// (histogram -> scan -> scatter, the bucket matrix of Sec. 3.4 (3)); each
// cell is then resolved once against the same cell of the frontier bucket:
// D = the cell's frontier (dst_h) ids, S = its sampled ids, new = S \ D.
// Tiles ascend in id, so new_h in ascending order is the cells' new ids in
// tile order, and a per-minibatch scan of the cells' new counts over tiles
// places every new node in src_h = dst_h ++ new_h.  Resolving a cell gives,
// with ranks local to the cell, each sampled edge's col and the cell of the
// next hop's frontier bucket (D | new in ascending id); after the scans, a
// fix-up pass and a compaction pass turn the local ranks into final indices.
// The bucket is carried from hop to hop and never rebuilt.  This file holds
// the scatter, the scans, the fix-up and the compaction, and the cell kernels
// of the sampled frontier; the default frontier's cells are resolved in
// dedup_cells.cu.
#include "common.cuh"
#include "internal.h"

namespace agnes {

namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kIlp = 4;  // independent elements per thread in the streaming passes

// Places every sampled edge of minibatch j at soff[cell] + rank (cell and
// rank were recorded while sampling), building the sampled bucket: (id, edge
// index) pairs, or packed 4-byte entries edge index << 12 | tile-local id.
__global__ void __launch_bounds__(kThreads)
dedup_scatter_kernel(const int32_t* __restrict__ nbr, const int32_t* __restrict__ ecnt,
                     int64_t ecap, const int32_t* __restrict__ scell,
                     const int32_t* __restrict__ srank, const int32_t* __restrict__ soff,
                     int2* __restrict__ sb, bool packed, const int32_t* status) {
  grid_dep_wait();
  if (failed(status)) return;
  const int32_t j = blockIdx.y;
  const int64_t E = ecnt[j];
  const int64_t o = (int64_t)j * ecap;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < E;
       e += (int64_t)gridDim.x * blockDim.x) {
    if (packed) {  // nbr holds rank << 12 | tile-local id; e < 2^20
      const uint32_t v = (uint32_t)nbr[o + e];
      reinterpret_cast<uint32_t*>(sb)[soff[scell[o + e]] + (v >> 12)] =
          ((uint32_t)e << 12) | (v & 0xfffu);
    } else {
      sb[soff[scell[o + e]] + srank[o + e]] = make_int2(nbr[o + e], (int32_t)e);
    }
  }
}

struct CellArgs {
  TileMap tm;
  int32_t H;
  int64_t ncells;
  int64_t capK, ecap;
  const int32_t* fb_id;      // frontier bucket (ids sorted inside a cell)
  const int32_t* fb_pos;
  const int32_t* fcell_off;
  const int2* sb;            // sampled bucket: (id, edge index)
  const int32_t* soff;
  const int32_t* tile_adj_block;
  uint8_t* adj_flags;
  int32_t* newcnt;           // per cell: new ids
  int32_t* nfcnt;            // per cell: next-frontier entries
  int2* tmp;                 // per cell at fcell_off + soff: next-frontier entries, local ranks
  int32_t* col;              // H x ecap: final col, or -(1 + local new rank)
  int32_t* big_list;         // cells with more than kDedupSmallMax entries
  int32_t* big_n;
  bool sampled;              // next frontier = the cell's distinct sampled ids
  const int32_t* status;
};

// A cell (t, j): its frontier entries [fo, fo+fn) and sampled entries
// [so, so+sn).
struct Cell {
  int32_t fo, fn, so, sn, t, j;
};

__device__ __forceinline__ bool load_cell(const CellArgs& a, int64_t cell, Cell* c) {
  if (cell >= a.ncells) {
    *c = Cell{0, 0, 0, 0, 0, 0};
    return false;
  }
  c->fo = a.fcell_off[cell];
  c->fn = a.fcell_off[cell + 1] - c->fo;
  c->so = a.soff[cell];
  c->sn = a.soff[cell + 1] - c->so;
  c->t = (int32_t)((uint32_t)cell / (uint32_t)a.H);  // cells < 2^31
  c->j = (int32_t)(cell - (int64_t)c->t * a.H);
  return true;
}

// ---- small cells: entry-parallel -----------------------------------------------
//
// A CTA takes 128 consecutive cells and stages the entries of the cells with
// samples and at most 32 entries in shared memory, each cell's frontier
// entries (sorted) followed by its sampled entries.  Every thread then
// resolves one entry against the entries of its own cell:
//   phase 1, sampled entry u: inD = u is a frontier id of the cell (binary
//            search) and which; leader = not inD and no earlier sampled entry
//            of the cell is u;
//   phase 2: lessN = leaders of the cell smaller than u, lessF = frontier ids
//            smaller than u (a frontier entry's own index); the entry's rank
//            in the next-frontier cell is lessF + lessN and a new node's rank
//            among the cell's new ids is lessN.
// Cells with more than 32 entries go to the big-cell list.
constexpr int kCellThreads = 128;  // threads per CTA of the cells kernel
constexpr int kCompactIlp = 2;     // bucket entries per thread and round of the compaction (4 and 8 measured slower)
constexpr int kGroupCells = kCellThreads;
constexpr int kSlotCap = 1024;
constexpr int kSmallMax = kDedupSmallMax;
constexpr int kRoundFill = kSlotCap - kSmallMax;  // a cell starting below this fits

enum : uint8_t { kSlotF = 1, kSlotLeader = 2, kSlotInD = 4, kSlotFirst = 8 };

struct GroupSmem {
  int32_t fn[kGroupCells];
  int32_t ps[kGroupCells + 1];  // staged-slot prefix of the group's cells
  int32_t tb[kGroupCells];      // tmp base of the cell
  int32_t j[kGroupCells];
  int32_t wsum[kCellThreads / 32];
  int32_t id[kSlotCap];
  int32_t x[kSlotCap];       // frontier: output row; sampled: edge index
  int16_t fidx[kSlotCap];    // sampled inD: slot of the matching frontier entry
  uint8_t cell[kSlotCap];
  uint8_t flag[kSlotCap];
};

__device__ __forceinline__ void put_tmp(const CellArgs& a, int32_t at, int32_t id, int32_t x) {
  a.tmp[at] = make_int2(id, x);
}

__global__ void __launch_bounds__(kCellThreads) dedup_cells_kernel(CellArgs a) {
  grid_dep_wait();
  if (failed(a.status)) return;
  __shared__ GroupSmem sm;
  const int tid = threadIdx.x, lane = lane_id(), warp = tid >> 5;
  const int64_t ngroups = (a.ncells + kGroupCells - 1) / kGroupCells;
  for (int64_t grp = blockIdx.x; grp < ngroups; grp += gridDim.x) {
    const int64_t c0 = grp * kGroupCells;
    const int64_t my_cell = c0 + tid;
    // per-cell facts, one thread per cell
    Cell c;
    const bool valid = load_cell(a, my_cell, &c);
    const int n = c.fn + c.sn;
    const bool staged = valid && c.sn > 0 && n <= kSmallMax;
    if (valid) {
      if (c.fn > 0) a.adj_flags[a.tile_adj_block[c.t]] = 1;
      if (n > kSmallMax) {
        a.big_list[atomicAdd(a.big_n, 1)] = (int32_t)my_cell;
      } else if (c.sn == 0) {
        a.newcnt[my_cell] = 0;
        a.nfcnt[my_cell] = a.sampled ? 0 : c.fn;
      }
    }
    const int32_t ns = staged ? n : 0;
    sm.fn[tid] = c.fn;
    sm.j[tid] = c.j;
    sm.tb[tid] = c.fo + c.so;
    const int32_t inc = warp_incl_scan(ns);
    if (lane == 31) sm.wsum[warp] = inc;
    __syncthreads();
    {
      int32_t off = 0, tot = 0;
      for (int w = 0; w < kCellThreads / 32; ++w) {
        off += w < warp ? sm.wsum[w] : 0;
        tot += sm.wsum[w];
      }
      sm.ps[tid] = off + inc - ns;
      if (tid == 0) sm.ps[kGroupCells] = tot;
    }
    __syncthreads();
    const int32_t total = sm.ps[kGroupCells];
    // rounds: each starts at a cell start and takes the cells that start less
    // than kRoundFill slots later (a cell has at most 32 entries, so a round
    // never needs more than kSlotCap slots)
    for (int32_t rbase = 0, rend = 0; rbase < total; rbase = rend) {
      int32_t lo = 0, hi = kGroupCells;  // first cell with ps >= rbase + kRoundFill
      while (lo < hi) {
        const int32_t mid = (lo + hi) >> 1;
        if (sm.ps[mid] < rbase + kRoundFill) lo = mid + 1; else hi = mid;
      }
      rend = min(total, sm.ps[lo]);  // slots [rbase, rend)
      const int32_t used = rend - rbase;
      const bool mine_in_round = staged && sm.ps[tid] >= rbase && sm.ps[tid] < rend;
      // the owner of each cell of the round maps its slots to the cell
      if (mine_in_round)
        for (int q = 0; q < n; ++q) sm.cell[sm.ps[tid] - rbase + q] = (uint8_t)tid;
      __syncthreads();
      for (int32_t sl = tid; sl < used; sl += kCellThreads) {
        const int l = sm.cell[sl];
        const int32_t q = rbase + sl - sm.ps[l];
        const int32_t fnl = sm.fn[l];
        // this cell's frontier / sampled entries start at tb - so / tb - fo
        if (q < fnl) {
          const int32_t fo = __ldg(a.fcell_off + c0 + l);
          sm.id[sl] = a.fb_id[fo + q];
          sm.x[sl] = a.fb_pos[fo + q];
          sm.flag[sl] = kSlotF;
        } else {
          const int32_t so = __ldg(a.soff + c0 + l);
          const int2 e = a.sb[so + q - fnl];
          sm.id[sl] = e.x;
          sm.x[sl] = e.y;
          sm.flag[sl] = 0;
        }
      }
      __syncthreads();
      // phase 1: membership and first occurrence of sampled ids
      for (int32_t sl = tid; sl < used; sl += kCellThreads) {
        if (sm.flag[sl] & kSlotF) continue;
        const int l = sm.cell[sl];
        const int32_t fs = sm.ps[l] - rbase, fe = fs + sm.fn[l];
        const int32_t id = sm.id[sl];
        int32_t lo2 = fs, hi2 = fe;  // first frontier id >= id (sorted)
        while (lo2 < hi2) {
          const int32_t mid = (lo2 + hi2) >> 1;
          if (sm.id[mid] < id) lo2 = mid + 1; else hi2 = mid;
        }
        uint8_t fl = 0;
        const bool inD = lo2 < fe && sm.id[lo2] == id;
        if (inD) {
          fl = kSlotInD;
          sm.fidx[sl] = (int16_t)lo2;
        }
        if (!inD || a.sampled) {  // first occurrence among the cell's samples
          bool dup = false;
          for (int32_t q = fe; q < sl; ++q) dup |= sm.id[q] == id;
          if (!dup) fl |= (inD ? 0 : kSlotLeader) | (a.sampled ? kSlotFirst : 0);
        }
        sm.flag[sl] = fl;
      }
      __syncthreads();
      // the owner counts its cell's new ids
      if (mine_in_round) {
        const int32_t fs = sm.ps[tid] - rbase;
        int32_t cnt = 0, first = 0;
        for (int32_t q = fs + c.fn; q < fs + n; ++q) {
          cnt += (sm.flag[q] & kSlotLeader) != 0;
          first += (sm.flag[q] & kSlotFirst) != 0;
        }
        a.newcnt[my_cell] = cnt;
        a.nfcnt[my_cell] = a.sampled ? first : c.fn + cnt;
      }
      // phase 2: local ranks, col, next-frontier entries
      for (int32_t sl = tid; sl < used; sl += kCellThreads) {
        const int l = sm.cell[sl];
        const int32_t fs = sm.ps[l] - rbase, fe = fs + sm.fn[l], se = sm.ps[l + 1] - rbase;
        const int32_t id = sm.id[sl];
        const uint8_t fl = sm.flag[sl];
        int32_t lessN = 0;
        for (int32_t q = fe; q < se; ++q) lessN += (sm.flag[q] & kSlotLeader) && sm.id[q] < id;
        const int32_t tb = sm.tb[l];
        if (fl & kSlotF) {
          if (!a.sampled) put_tmp(a, tb + (sl - fs) + lessN, id, sm.x[sl]);
          continue;
        }
        if (fl & kSlotFirst) {  // sampled frontier: the cell's distinct samples, ascending
          int32_t lessS = 0;
          for (int32_t q = fe; q < se; ++q) lessS += (sm.flag[q] & kSlotFirst) && sm.id[q] < id;
          put_tmp(a, tb + lessS, id, 0);
        }
        const int64_t jrow = (int64_t)sm.j[l] * a.ecap;
        if (fl & kSlotInD) {
          a.col[jrow + sm.x[sl]] = (int32_t)(sm.x[sm.fidx[sl]] - (int64_t)sm.j[l] * a.capK);
          continue;
        }
        a.col[jrow + sm.x[sl]] = -1 - lessN;
        if ((fl & kSlotLeader) && !a.sampled) {
          int32_t lo2 = fs, hi2 = fe;  // frontier ids smaller than id
          while (lo2 < hi2) {
            const int32_t mid = (lo2 + hi2) >> 1;
            if (sm.id[mid] < id) lo2 = mid + 1; else hi2 = mid;
          }
          put_tmp(a, tb + (lo2 - fs) + lessN, id, -1 - lessN);
        }
      }
      __syncthreads();
    }
  }
}

// ---- big cells: one warp each, bitmaps over the tile ---------------------------

__device__ __forceinline__ void mark_bits(const CellArgs& a, const Cell& c, uint32_t* D,
                                          uint32_t* S, int32_t base, int32_t words) {
  const int lane = lane_id();
  for (int w = lane; w < words; w += 32) {
    D[w] = 0;
    S[w] = 0;
  }
  __syncwarp();
  for (int32_t i0 = lane; i0 < c.fn; i0 += 128) {  // four entries in flight per lane
    int32_t v[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) v[q] = i0 + 32 * q < c.fn ? a.fb_id[c.fo + i0 + 32 * q] - base : -1;
#pragma unroll
    for (int q = 0; q < 4; ++q)
      if (v[q] >= 0) atomicOr(&D[v[q] >> 5], 1u << (v[q] & 31));
  }
  for (int32_t i0 = lane; i0 < c.sn; i0 += 128) {
    int32_t v[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) v[q] = i0 + 32 * q < c.sn ? a.sb[c.so + i0 + 32 * q].x - base : -1;
#pragma unroll
    for (int q = 0; q < 4; ++q)
      if (v[q] >= 0) atomicOr(&S[v[q] >> 5], 1u << (v[q] & 31));
  }
  __syncwarp();
}

__global__ void __launch_bounds__(kThreads) dedup_big_kernel(CellArgs a) {
  grid_dep_wait();
  if (failed(a.status)) return;
  __shared__ uint32_t D_s[kWarps][kTileWords];
  __shared__ uint32_t N_s[kWarps][kTileWords];
  __shared__ int32_t pD_s[kWarps][kTileWords];
  __shared__ int32_t pN_s[kWarps][kTileWords];
  const int warp = threadIdx.x >> 5, lane = lane_id();
  uint32_t* D = D_s[warp];
  uint32_t* Nw = N_s[warp];
  int32_t* pD = pD_s[warp];
  int32_t* pN = pN_s[warp];
  const int32_t nbig = *a.big_n;
  const int64_t nwarps = (int64_t)gridDim.x * kWarps;
  for (int64_t b = blockIdx.x * (int64_t)kWarps + warp; b < nbig; b += nwarps) {
    const int64_t cell = a.big_list[b];
    Cell c;
    load_cell(a, cell, &c);
    if (c.sn == 0) {  // nothing sampled: the compaction copies the frontier cell
      if (lane == 0) {
        a.newcnt[cell] = 0;
        a.nfcnt[cell] = a.sampled ? 0 : c.fn;
      }
      continue;
    }
    const int32_t base = a.tm.tile_first[c.t];
    const int32_t words = (a.tm.tile_first[c.t + 1] - base + 31) >> 5;
    mark_bits(a, c, D, Nw, base, words);
    // new = S & ~D; per-word exclusive ranks of D and new
    uint32_t dw[4], nw[4], sw[4];
    int32_t sd = 0, snw = 0, ssw = 0;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int w = lane * 4 + q;
      dw[q] = w < words ? D[w] : 0u;
      sw[q] = w < words ? Nw[w] : 0u;
      nw[q] = sw[q] & ~dw[q];
      sd += __popc(dw[q]);
      snw += __popc(nw[q]);
      ssw += __popc(sw[q]);
    }
    const int32_t tot_new = warp_sum(snw);
    const int32_t tot_s = warp_sum(ssw);
    int32_t rd = warp_incl_scan(sd) - sd;
    int32_t rn = warp_incl_scan(snw) - snw;
    int32_t rs = warp_incl_scan(ssw) - ssw;
    __syncwarp();
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int w = lane * 4 + q;
      Nw[w] = nw[q];
      pD[w] = rd;
      pN[w] = rn;
      rd += __popc(dw[q]);
      rn += __popc(nw[q]);
    }
    __syncwarp();
    if (lane == 0) {
      a.newcnt[cell] = tot_new;
      a.nfcnt[cell] = a.sampled ? tot_s : c.fn + tot_new;
    }
    const int64_t jcap = (int64_t)c.j * a.capK;
    int32_t* col = a.col + (int64_t)c.j * a.ecap;
    for (int32_t i = lane; i < c.sn; i += 32) {
      const int2 se = a.sb[c.so + i];
      const int32_t lu = se.x - base;
      const int32_t w = lu >> 5;
      const uint32_t bit = 1u << (lu & 31), below = bit - 1u;
      col[se.y] = (D[w] & bit) ? (int32_t)(a.fb_pos[c.fo + pD[w] + __popc(D[w] & below)] - jcap)
                               : -1 - (pN[w] + __popc(Nw[w] & below));
    }
    const int32_t tb = c.fo + c.so;
    if (a.sampled) {  // the tile's distinct sampled ids, ascending
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int w = lane * 4 + q;
        uint32_t rest = w < words ? sw[q] : 0u;
        while (rest) {
          const int bb = __ffs(rest) - 1;
          rest &= rest - 1u;
          put_tmp(a, tb + rs + __popc(sw[q] & ((1u << bb) - 1u)), base + w * 32 + bb, 0);
        }
        rs += __popc(sw[q]);
      }
      __syncwarp();
      continue;
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int w = lane * 4 + q;
      if (w >= words) break;
      const uint32_t d = dw[q], nn = nw[q];
      uint32_t rest = d | nn;
      const int32_t r0 = pD[w] + pN[w];
      while (rest) {
        const int bb = __ffs(rest) - 1;
        rest &= rest - 1u;
        const uint32_t below = (1u << bb) - 1u;
        const int32_t id = base + w * 32 + bb;
        const int32_t r = r0 + __popc((d | nn) & below);
        const int32_t x = ((d >> bb) & 1u) ? a.fb_pos[c.fo + pD[w] + __popc(d & below)]
                                           : -1 - (pN[w] + __popc(nn & below));
        put_tmp(a, tb + r, id, x);
      }
    }
    __syncwarp();
  }
}

// ---- fix-up and compaction (after the scans) --------------------------------------

// col[e] = -(1 + r) becomes the new node's index in src_h:
// |dst_h| + (new ids of the minibatch in earlier tiles) + r.
__global__ void __launch_bounds__(kThreads)
dedup_fix_col_kernel(int32_t* __restrict__ col, const int32_t* __restrict__ ecnt, int64_t ecap,
                     const int32_t* __restrict__ scell, const int32_t* __restrict__ newbase,
                     const int32_t* __restrict__ nsz_prev, const int32_t* status) {
  grid_dep_wait();
  if (failed(status)) return;
  const int32_t j = blockIdx.y;
  const int64_t E = ecnt[j];
  const int64_t o = (int64_t)j * ecap;
  const int32_t base = nsz_prev[j];
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t e0 = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e0 < E;
       e0 += kIlp * stride) {  // kIlp edges per thread: their base loads in flight together
    int32_t v[kIlp], cell[kIlp], nb[kIlp];
#pragma unroll
    for (int k = 0; k < kIlp; ++k) {
      const int64_t e = e0 + k * stride;
      v[k] = e < E ? col[o + e] : 0;
      cell[k] = e < E ? scell[o + e] : 0;
    }
#pragma unroll
    for (int k = 0; k < kIlp; ++k) nb[k] = v[k] < 0 ? newbase[cell[k]] : 0;
#pragma unroll
    for (int k = 0; k < kIlp; ++k)
      if (v[k] < 0) col[o + e0 + k * stride] = base + nb[k] + (-1 - v[k]);
  }
}

struct CompactArgs {
  int64_t ncells;
  int32_t H;
  int64_t capK;
  const int32_t* fb_id;
  const int32_t* fb_pos;
  const int32_t* fcell_off;
  const int32_t* soff;
  const int2* tmp;
  const int32_t* nfcell_off;
  const int32_t* newbase;
  const int32_t* nsz_prev;
  const int32_t* noutbase;   // sampled frontier: rows are positions among the distinct samples
  bool sampled;
  int32_t* nfb_id;
  int32_t* nfb_pos;
  int32_t* nodes;
  const int32_t* status;
};

// Writes the next frontier bucket in cell order: a cell without samples is
// copied from the current bucket, any other from its tmp entries, where a new
// node (x = -(1 + r)) gets its output row j * capK + |dst_h| + newbase + r and
// its id is appended to the minibatch's node list.
__global__ void __launch_bounds__(kCellThreads) dedup_compact_kernel(CompactArgs a) {
  grid_dep_wait();
  if (failed(a.status)) return;
  __shared__ int32_t s_nfo[kGroupCells + 1];
  __shared__ int32_t s_src[kGroupCells];   // source base in fb (>= 0) or ~base in tmp
  __shared__ int32_t s_row[kGroupCells];   // j * capK + |dst_h| + newbase
  const int tid = threadIdx.x;
  const int64_t ngroups = (a.ncells + kGroupCells - 1) / kGroupCells;
  for (int64_t grp = blockIdx.x; grp < ngroups; grp += gridDim.x) {
    const int64_t c0 = grp * kGroupCells;
    const int64_t cell = c0 + tid;
    const int64_t last = min(a.ncells, c0 + kGroupCells);
    if (cell < a.ncells) {
      const int32_t fo = a.fcell_off[cell];
      const int32_t so = a.soff[cell];
      const int32_t sn = a.soff[cell + 1] - so;
      const int32_t j = (int32_t)((uint32_t)cell % (uint32_t)a.H);
      s_nfo[tid] = a.nfcell_off[cell];
      s_src[tid] = sn == 0 && !a.sampled ? fo : ~(fo + so);
      s_row[tid] = (int32_t)((int64_t)j * a.capK +
                             (a.sampled ? a.noutbase[cell] : a.nsz_prev[j] + a.newbase[cell]));
    }
    if (tid == 0) s_nfo[last - c0] = a.nfcell_off[last];
    __syncthreads();
    const int32_t k0 = s_nfo[0], k1 = s_nfo[last - c0];
    // kCompactIlp entries per thread and round: their loads in flight before the stores
    for (int32_t kb = k0 + tid; kb < k1; kb += kCompactIlp * kCellThreads) {
      int32_t cl[kCompactIlp], r[kCompactIlp], id[kCompactIlp], pos[kCompactIlp];
      bool in[kCompactIlp];
#pragma unroll
      for (int u = 0; u < kCompactIlp; ++u) {
        const int32_t k = kb + u * kCellThreads;
        in[u] = k < k1;
        int32_t lo = 0, hi = (int32_t)(last - c0);  // last cell with nfo <= k
        while (hi - lo > 1) {
          const int32_t mid = (lo + hi) >> 1;
          if (s_nfo[mid] <= k) lo = mid; else hi = mid;
        }
        cl[u] = lo;
        r[u] = k - s_nfo[lo];
        id[u] = 0;
        pos[u] = 0;
        if (in[u]) {
          const int32_t src = s_src[lo];
          if (src >= 0) {
            id[u] = a.fb_id[src + r[u]];
            pos[u] = a.fb_pos[src + r[u]];
          } else {
            const int2 e = a.tmp[~src + r[u]];
            id[u] = e.x;
            pos[u] = e.y;
          }
        }
      }
#pragma unroll
      for (int u = 0; u < kCompactIlp; ++u) {
        if (!in[u]) continue;
        const int32_t k = kb + u * kCellThreads;
        if (s_src[cl[u]] < 0) {
          if (a.sampled) {
            pos[u] = s_row[cl[u]] + r[u];
            a.nodes[pos[u]] = id[u];
          } else if (pos[u] < 0) {
            pos[u] = s_row[cl[u]] + (-1 - pos[u]);
            a.nodes[pos[u]] = id[u];
          }
        }
        a.nfb_id[k] = id[u];
        a.nfb_pos[k] = pos[u];
      }
    }
    __syncthreads();
  }
}

}  // namespace

cudaError_t launch_dedup(const HopArgs& a, const DedupBufs& d, int num_sms, cudaStream_t st) {
  const TileMap tm{a.tile_first, a.chunk_tile, a.T};
  const int64_t ncells = (int64_t)a.T * a.H;
  int gx = (num_sms * 8 + a.H - 1) / a.H;
  if (gx < 1) gx = 1;
  const dim3 egrid(gx, a.H);
  cudaError_t e = cells_scan(d.scnt, d.soff, ncells, d.flat_scratch, d.scan_scratch, a.status, st);
  if (e != cudaSuccess) return e;
  dedup_scatter_kernel<<<egrid, kThreads, 0, st>>>(d.nbr, d.ecnt, a.ecap, d.scell, d.srank,
                                                   d.soff, d.sb, a.sb_packed, a.status);

  CellArgs c;
  c.tm = tm;
  c.H = a.H;
  c.ncells = ncells;
  c.capK = a.capK;
  c.ecap = a.ecap;
  c.fb_id = d.fb_id;
  c.fb_pos = d.fb_pos;
  c.fcell_off = d.fcell_off;
  c.sb = d.sb;
  c.soff = d.soff;
  c.tile_adj_block = d.tile_adj_block;
  c.adj_flags = d.adj_flags;
  c.newcnt = d.newcnt;
  c.nfcnt = d.nfcnt;
  c.tmp = d.tmp;
  c.col = d.col;
  c.big_list = d.big_list;
  c.big_n = d.big_n;
  c.sampled = d.frontier_sampled;
  c.status = a.status;
  if (d.frontier_sampled) {
    if ((e = cudaMemsetAsync(d.big_n, 0, sizeof(int32_t), st)) != cudaSuccess) return e;
    dedup_cells_kernel<<<resident_grid((const void*)dedup_cells_kernel, kCellThreads, num_sms),
                         kCellThreads, 0, st>>>(c);
    dedup_big_kernel<<<resident_grid((const void*)dedup_big_kernel, kThreads, num_sms), kThreads,
                       0, st>>>(c);
  } else {
    e = launch_dedup_cells(a, d, num_sms, st);  // dedup_cells.cu
    if (e != cudaSuccess) return e;
  }
  // per-minibatch offsets of the new ids: scan down the tiles of the
  // tile-major [T x H] count matrix; totals give the next frontier sizes
  // |src_h| = |dst_h| + new ids; the next frontier is src_h, or (sampled
  // frontier) the distinct sampled ids, numbered by their own column scan.
  // With a side stream, the new-id scan and the col fix-up (which needs only
  // its result) run there, beside the scans of the next-frontier counts; the
  // side stream has its own scan scratch, and the compaction waits for the
  // new-id offsets.
  cudaStream_t nst = st;
  int64_t* nscratch = d.scan_scratch;
  if (d.side) {
    if ((e = cudaEventRecord(d.fork, st)) != cudaSuccess) return e;
    if ((e = cudaStreamWaitEvent(d.side, d.fork, 0)) != cudaSuccess) return e;
    nst = d.side;
    nscratch = d.side_scratch;
  }
  e = col_scan(d.newcnt, d.newbase, a.T, a.H, d.nsz_prev, d.srcsz, nscratch, a.status, nst);
  if (e != cudaSuccess) return e;
  if (d.side && (e = cudaEventRecord(d.ready, d.side)) != cudaSuccess) return e;
  dedup_fix_col_kernel<<<egrid, kThreads, 0, nst>>>(d.col, d.ecnt, a.ecap, d.scell, d.newbase,
                                                    d.nsz_prev, a.status);
  if (d.frontier_sampled) {
    e = col_scan(d.nfcnt, d.noutbase, a.T, a.H, nullptr, d.nsz_next, d.scan_scratch, a.status,
                 st);
    if (e != cudaSuccess) return e;
  }
  e = cells_scan(d.nfcnt, d.nfcell_off, ncells, d.flat_scratch, d.scan_scratch, a.status, st);
  if (e != cudaSuccess) return e;
  if (d.side && (e = cudaStreamWaitEvent(st, d.ready, 0)) != cudaSuccess) return e;
  if (!d.frontier_sampled) {
    e = cudaMemcpyAsync(d.nsz_next, d.srcsz, sizeof(int32_t) * a.H, cudaMemcpyDeviceToDevice, st);
    if (e != cudaSuccess) return e;
  }
  return cudaGetLastError();
}

cudaError_t launch_dedup_compact(const HopArgs& a, const DedupBufs& d, int num_sms,
                                 cudaStream_t st) {
  const int64_t ncells = (int64_t)a.T * a.H;
  CompactArgs k;
  k.ncells = ncells;
  k.H = a.H;
  k.capK = a.capK;
  k.fb_id = d.fb_id;
  k.fb_pos = d.fb_pos;
  k.fcell_off = d.fcell_off;
  k.soff = d.soff;
  k.tmp = d.tmp;
  k.nfcell_off = d.nfcell_off;
  k.newbase = d.newbase;
  k.nsz_prev = d.nsz_prev;
  k.noutbase = d.noutbase;
  k.sampled = d.frontier_sampled;
  k.nfb_id = d.nfb_id;
  k.nfb_pos = d.nfb_pos;
  k.nodes = d.nodes;
  k.status = a.status;
  dedup_compact_kernel<<<resident_grid((const void*)dedup_compact_kernel, kCellThreads, num_sms),
                         kCellThreads, 0, st>>>(k);
  return cudaGetLastError();
}

}  // namespace agnes
