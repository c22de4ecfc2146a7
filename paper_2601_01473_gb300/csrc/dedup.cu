// dedup.cu -- per-minibatch union / dedup and relabelling of a hop's samples
// (Algorithm 1: N^j_out <- N^j_out u Sample(j, ...), N_in <- N_out).
//
// The sampled ids of every minibatch are bucketed by (tile, minibatch) cell
// (histogram -> scan -> scatter, the bucket matrix of Sec. 3.4 (3)).  A cell
// covers at most 4096 consecutive ids, so one warp resolves it with two
// shared-memory bitmaps over the tile: D = the cell's frontier (dst_h) ids and
// S = its sampled ids.  new = S & ~D in ascending id order is the cell's part
// of new_h (tiles ascend in id, so a per-minibatch scan of the cells' new
// counts over tiles gives each new node its index in src_h = dst_h ++ new_h);
// popcount ranks in D and new give every sampled edge its col; and D | new in
// ascending order, with each node's output row, is the cell of the next hop's
// frontier bucket -- the bucket is carried from hop to hop and never rebuilt.
#include "common.cuh"
#include "internal.h"

namespace agnes {

namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;

// Places every sampled edge of minibatch j at soff[cell] + rank (cell and
// rank were recorded while sampling), building the sampled bucket.
__global__ void __launch_bounds__(kThreads)
dedup_scatter_kernel(const int32_t* __restrict__ nbr, const int32_t* __restrict__ ecnt,
                     int64_t ecap, const int32_t* __restrict__ scell,
                     const int32_t* __restrict__ srank, const int32_t* __restrict__ soff,
                     int2* __restrict__ sb, const int32_t* status) {
  if (failed(status)) return;
  const int32_t j = blockIdx.y;
  const int64_t E = ecnt[j];
  const int64_t o = (int64_t)j * ecap;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < E;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int32_t slot = soff[scell[o + e]] + srank[o + e];
    sb[slot] = make_int2(nbr[o + e], (int32_t)e);
  }
}

struct CellArgs {
  TileMap tm;
  int32_t H;
  int64_t ncells;
  int64_t capK, ecap;
  const int32_t* fb_id;
  const int32_t* fb_pos;
  const int32_t* fcell_off;
  const int2* sb;        // sampled bucket: (id, edge index) per slot
  const int32_t* soff;
  int32_t* big_list;     // cells with more than 32 entries
  int32_t* big_n;
  const int32_t* tile_adj_block;
  uint8_t* adj_flags;
  int32_t* newcnt;
  const int32_t* newbase;
  int32_t* nfcnt;
  const int32_t* nfcell_off;
  int32_t* nfb_id;
  int32_t* nfb_pos;
  const int32_t* nsz_prev;
  int32_t* nodes;
  int32_t* col;
  const int32_t* status;
};

// Marks the cell's frontier ids in D and sampled ids in S (tile-local bits).
__device__ __forceinline__ void mark_cell(const CellArgs& a, uint32_t* D, uint32_t* S, int32_t base,
                                          int32_t words, int32_t fo, int32_t fn, int32_t so,
                                          int32_t sn) {
  const int lane = lane_id();
  for (int w = lane; w < words; w += 32) {
    D[w] = 0;
    S[w] = 0;
  }
  __syncwarp();
  // four entries in flight per lane
  for (int32_t i0 = lane; i0 < fn; i0 += 128) {
    int32_t v[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) v[q] = i0 + 32 * q < fn ? a.fb_id[fo + i0 + 32 * q] - base : -1;
#pragma unroll
    for (int q = 0; q < 4; ++q)
      if (v[q] >= 0) atomicOr(&D[v[q] >> 5], 1u << (v[q] & 31));
  }
  for (int32_t i0 = lane; i0 < sn; i0 += 128) {
    int32_t v[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) v[q] = i0 + 32 * q < sn ? a.sb[so + i0 + 32 * q].x - base : -1;
#pragma unroll
    for (int q = 0; q < 4; ++q)
      if (v[q] >= 0) atomicOr(&S[v[q] >> 5], 1u << (v[q] & 31));
  }
  __syncwarp();
}

// A cell (t, j): its frontier entries [fo, fo+fn) and sampled entries
// [so, so+sn).
struct Cell {
  int32_t fo, fn, so, sn, t, j;
};

// Loads the cell of this lane (one cell per lane, 32 consecutive cells per
// warp); returns false past the last cell.
__device__ __forceinline__ bool load_cell(const CellArgs& a, int64_t cell, Cell* c) {
  if (cell >= a.ncells) {
    *c = Cell{0, 0, 0, 0, 0, 0};
    return false;
  }
  c->fo = a.fcell_off[cell];
  c->fn = a.fcell_off[cell + 1] - c->fo;
  c->so = a.soff[cell];
  c->sn = a.soff[cell + 1] - c->so;
  c->t = (int32_t)(cell / a.H);
  c->j = (int32_t)(cell - (int64_t)c->t * a.H);
  return true;
}

__device__ __forceinline__ Cell bcast(const Cell& c, int k) {
  Cell o;
  o.fo = __shfl_sync(0xffffffffu, c.fo, k);
  o.fn = __shfl_sync(0xffffffffu, c.fn, k);
  o.so = __shfl_sync(0xffffffffu, c.so, k);
  o.sn = __shfl_sync(0xffffffffu, c.sn, k);
  o.t = __shfl_sync(0xffffffffu, c.t, k);
  o.j = __shfl_sync(0xffffffffu, c.j, k);
  return o;
}

// Small cells (at most 32 entries) are packed several to a warp pass: the
// cells of the pass take consecutive lanes (cell r owns lanes
// [start_r, start_r + n_r)), one entry per lane, frontier entries first.
// Equal ids of one cell are found with match_any on (r, id); ranks are
// counted against the other lanes of the same cell.
struct Pass {
  unsigned cells;  // lanes (of the 32-cell chunk) whose cell is in this pass
  int used;        // entry lanes used
};

struct Slot {
  bool act, isF, inD, leader;
  int r, cl;        // rank of the slot's cell in the pass, lane owning it
  int32_t id;
  int32_t extra;    // frontier: output row; sampled: edge index
  unsigned long long key;
  unsigned peers, fm, lm;
  Cell c;
};

// Chooses the next pass among the remaining small cells (in lane order, as
// many as fit in 32 lanes); returns this lane's first entry lane in *start.
__device__ __forceinline__ Pass next_pass(unsigned* remaining, int n, int* start) {
  const int lane = lane_id();
  const bool rem = (*remaining >> lane) & 1u;
  const int mine = rem ? n : 0;
  const int incl = warp_incl_scan(mine);
  const bool fits = rem && incl <= 32;
  Pass p;
  p.cells = __ballot_sync(0xffffffffu, fits);
  p.used = __shfl_sync(0xffffffffu, incl, 31 - __clz(p.cells));
  *remaining &= ~p.cells;
  *start = incl - mine;
  return p;
}

__device__ __forceinline__ Slot load_slot(const CellArgs& a, const Pass& p, const Cell& mine,
                                          int start, int* cell_lane) {
  const int lane = lane_id();
  const bool in_pass = (p.cells >> lane) & 1u;
  if (in_pass) cell_lane[__popc(p.cells & ((1u << lane) - 1u))] = lane;
  __syncwarp();
  const unsigned starts = __reduce_or_sync(0xffffffffu, in_pass ? (1u << start) : 0u);
  Slot s;
  s.act = lane < p.used;
  s.r = s.act ? __popc(starts & ((2u << lane) - 1u)) - 1 : 0;
  s.cl = s.act ? cell_lane[s.r] : 0;
  __syncwarp();
  s.c = bcast(mine, s.cl);
  const int st = __shfl_sync(0xffffffffu, start, s.cl);
  const int q = lane - st;
  s.isF = s.act && q < s.c.fn;
  s.id = 0;
  s.extra = 0;
  if (s.act) {
    if (s.isF) {
      s.id = a.fb_id[s.c.fo + q];
      s.extra = a.fb_pos[s.c.fo + q];
    } else {
      const int2 e = a.sb[s.c.so + q - s.c.fn];
      s.id = e.x;
      s.extra = e.y;
    }
  }
  s.key = s.act ? (((unsigned long long)s.r << 32) | (uint32_t)s.id)
                : (0xffffffff00000000ull | (unsigned)lane);
  s.peers = __match_any_sync(0xffffffffu, s.key);
  s.fm = __ballot_sync(0xffffffffu, s.isF);
  s.inD = (s.peers & s.fm) != 0;
  s.leader = s.act && !s.isF && !s.inD && lane == __ffs(s.peers) - 1;
  s.lm = __ballot_sync(0xffffffffu, s.leader);
  return s;
}

// Lanes [start, start + n) as a mask (n <= 32).
__device__ __forceinline__ unsigned lane_range(int start, int n) {
  return n >= 32 ? 0xffffffffu : (((1u << n) - 1u) << start);
}

// Cells with more than 32 entries: bitmaps over the tile.
__device__ __forceinline__ int32_t big_count(const CellArgs& a, const Cell& c, uint32_t* D,
                                             uint32_t* S) {
  const int32_t base = a.tm.tile_first[c.t];
  const int32_t words = (a.tm.tile_first[c.t + 1] - base + 31) >> 5;
  mark_cell(a, D, S, base, words, c.fo, c.fn, c.so, c.sn);
  int32_t cnt = 0;
  for (int w = lane_id(); w < words; w += 32) cnt += __popc(S[w] & ~D[w]);
  cnt = warp_sum(cnt);
  __syncwarp();
  return cnt;
}

__global__ void __launch_bounds__(kThreads) dedup_count_kernel(CellArgs a) {
  if (failed(a.status)) return;
  const int warp = threadIdx.x >> 5, lane = lane_id();
  const int64_t nchunks = (a.ncells + 31) / 32;
  const int64_t nwarps = (int64_t)gridDim.x * kWarps;
  __shared__ int cell_lane_s[kWarps][32];
  for (int64_t ch = blockIdx.x * (int64_t)kWarps + warp; ch < nchunks; ch += nwarps) {
    const int64_t my_cell = ch * 32 + lane;
    Cell mine;
    const bool valid = load_cell(a, my_cell, &mine);
    const int n = mine.fn + mine.sn;
    int32_t my_cnt = 0;
    // cells with more than 32 entries go to the big-cell list (one warp each
    // in the next kernel, so a hub tile's cells spread over the GPU)
    const bool big = valid && n > 32;
    const unsigned bm = __ballot_sync(0xffffffffu, big);
    if (bm) {
      int32_t base = 0;
      if (lane == __ffs(bm) - 1) base = atomicAdd(a.big_n, __popc(bm));
      base = __shfl_sync(0xffffffffu, base, __ffs(bm) - 1);
      if (big) a.big_list[base + __popc(bm & ((1u << lane) - 1u))] = (int32_t)my_cell;
    }
    // small cells, packed
    unsigned remaining = __ballot_sync(0xffffffffu, valid && mine.sn > 0 && n <= 32);
    while (remaining) {
      int start;
      const Pass p = next_pass(&remaining, n, &start);
      const Slot sl = load_slot(a, p, mine, start, cell_lane_s[warp]);
      if ((p.cells >> lane) & 1u) my_cnt = __popc(sl.lm & lane_range(start, n));
    }
    if (valid && !big) {
      a.newcnt[(int64_t)mine.j * a.tm.T + mine.t] = my_cnt;
      a.nfcnt[my_cell] = mine.fn + my_cnt;
    }
    if (valid && mine.fn > 0) a.adj_flags[a.tile_adj_block[mine.t]] = 1;
  }
}

// One warp per big cell (listed by dedup_count_kernel).
__global__ void __launch_bounds__(kThreads) dedup_count_big_kernel(CellArgs a) {
  if (failed(a.status)) return;
  __shared__ uint32_t D_s[kWarps][kTileWords];
  __shared__ uint32_t S_s[kWarps][kTileWords];
  const int warp = threadIdx.x >> 5, lane = lane_id();
  const int32_t nbig = *a.big_n;
  const int64_t nwarps = (int64_t)gridDim.x * kWarps;
  for (int64_t b = blockIdx.x * (int64_t)kWarps + warp; b < nbig; b += nwarps) {
    const int64_t cell = a.big_list[b];
    Cell c;
    load_cell(a, cell, &c);
    const int32_t cnt = c.sn > 0 ? big_count(a, c, D_s[warp], S_s[warp]) : 0;
    if (lane == 0) {
      a.newcnt[(int64_t)c.j * a.tm.T + c.t] = cnt;
      a.nfcnt[cell] = c.fn + cnt;
    }
  }
}

// Emits a pass of small cells: col of every sampled entry, the new nodes
// (ascending, after the cell's new base nb), and the next frontier cell
// (frontier and new ids merged in ascending order at nfo).
__device__ __forceinline__ void small_emit(const CellArgs& a, const Pass& p, const Slot& s,
                                           int32_t my_nb, int32_t my_nfo) {
  const int32_t nb = __shfl_sync(0xffffffffu, my_nb, s.cl);
  const int32_t nfo = __shfl_sync(0xffffffffu, my_nfo, s.cl);
  int32_t lessF = 0, lessN = 0;
  for (int k = 0; k < p.used; ++k) {
    const unsigned long long kk = __shfl_sync(0xffffffffu, s.key, k);
    if ((kk >> 32) == (s.key >> 32) && (uint32_t)kk < (uint32_t)s.id) {
      lessF += (s.fm >> k) & 1u;
      lessN += (s.lm >> k) & 1u;
    }
  }
  const int lane = lane_id();
  const int src = s.inD ? __ffs(s.peers & s.fm) - 1 : lane;
  const int32_t fpos = __shfl_sync(0xffffffffu, s.extra, src);
  const int64_t jcap = (int64_t)s.c.j * a.capK;
  if (s.act && !s.isF)
    a.col[(int64_t)s.c.j * a.ecap + s.extra] = s.inD ? (int32_t)(fpos - jcap) : nb + lessN;
  if (s.act && (s.isF || s.leader)) {
    const int32_t r = nfo + lessF + lessN;
    int32_t g = s.extra;
    if (s.leader) {
      g = (int32_t)(jcap + nb + lessN);
      a.nodes[g] = s.id;
    }
    a.nfb_id[r] = s.id;
    a.nfb_pos[r] = g;
  }
}

__device__ __forceinline__ void big_emit(const CellArgs& a, const Cell& c, int32_t nb, int32_t nfo,
                                         uint32_t* D, uint32_t* Nw, int32_t* pD, int32_t* pN) {
  const int lane = lane_id();
  const int32_t base = a.tm.tile_first[c.t];
  const int32_t words = (a.tm.tile_first[c.t + 1] - base + 31) >> 5;
  mark_cell(a, D, Nw, base, words, c.fo, c.fn, c.so, c.sn);
  // new = S & ~D; per-word exclusive ranks of D and new
  uint32_t dw[4], nw[4];
  int32_t sd = 0, sn_ = 0;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int w = lane * 4 + q;
    dw[q] = w < words ? D[w] : 0u;
    nw[q] = w < words ? (Nw[w] & ~dw[q]) : 0u;
    sd += __popc(dw[q]);
    sn_ += __popc(nw[q]);
  }
  int32_t rd = warp_incl_scan(sd) - sd;
  int32_t rn = warp_incl_scan(sn_) - sn_;
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

  const int64_t jcap = (int64_t)c.j * a.capK;
  int32_t* col = a.col + (int64_t)c.j * a.ecap;
  for (int32_t i = lane; i < c.sn; i += 32) {
    const int2 se = a.sb[c.so + i];
    const int32_t lu = se.x - base;
    const int32_t w = lu >> 5;
    const uint32_t bit = 1u << (lu & 31), below = bit - 1u;
    int32_t cv;
    if (D[w] & bit)
      cv = (int32_t)(a.fb_pos[c.fo + pD[w] + __popc(D[w] & below)] - jcap);
    else
      cv = nb + pN[w] + __popc(Nw[w] & below);
    col[se.y] = cv;
  }
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int w = lane * 4 + q;
    if (w >= words) break;
    const uint32_t d = dw[q], n = nw[q];
    uint32_t rest = d | n;
    const int32_t r0 = pD[w] + pN[w];
    while (rest) {
      const int b = __ffs(rest) - 1;
      rest &= rest - 1u;
      const uint32_t below = (1u << b) - 1u;
      const int32_t id = base + w * 32 + b;
      const int32_t r = r0 + __popc((d | n) & below);
      int32_t g;
      if ((d >> b) & 1u) {
        g = a.fb_pos[c.fo + pD[w] + __popc(d & below)];
      } else {
        g = (int32_t)(jcap + nb + pN[w] + __popc(n & below));
        a.nodes[g] = id;
      }
      a.nfb_id[nfo + r] = id;
      a.nfb_pos[nfo + r] = g;
    }
  }
  __syncwarp();
}

__global__ void __launch_bounds__(kThreads) dedup_emit_kernel(CellArgs a) {
  if (failed(a.status)) return;
  __shared__ int cell_lane_s[kWarps][32];
  const int warp = threadIdx.x >> 5, lane = lane_id();
  const int64_t nchunks = (a.ncells + 31) / 32;
  const int64_t nwarps = (int64_t)gridDim.x * kWarps;
  for (int64_t ch = blockIdx.x * (int64_t)kWarps + warp; ch < nchunks; ch += nwarps) {
    const int64_t my_cell = ch * 32 + lane;
    Cell mine;
    const bool valid = load_cell(a, my_cell, &mine);
    const int n = mine.fn + mine.sn;
    int32_t my_nfo = 0, my_nb = 0;
    if (valid && n > 0 && n <= 32) {
      my_nfo = a.nfcell_off[my_cell];
      if (mine.sn > 0) my_nb = a.nsz_prev[mine.j] + a.newbase[(int64_t)mine.j * a.tm.T + mine.t];
    }
    // small cells (including frontier-only ones), packed
    unsigned remaining = __ballot_sync(0xffffffffu, valid && n > 0 && n <= 32);
    while (remaining) {
      int start;
      const Pass p = next_pass(&remaining, n, &start);
      const Slot sl = load_slot(a, p, mine, start, cell_lane_s[warp]);
      small_emit(a, p, sl, my_nb, my_nfo);
    }
  }
}

// One warp per big cell (the list built by dedup_count_kernel).
__global__ void __launch_bounds__(kThreads) dedup_emit_big_kernel(CellArgs a) {
  if (failed(a.status)) return;
  __shared__ uint32_t D_s[kWarps][kTileWords];
  __shared__ uint32_t N_s[kWarps][kTileWords];
  __shared__ int32_t pD_s[kWarps][kTileWords];
  __shared__ int32_t pN_s[kWarps][kTileWords];
  const int warp = threadIdx.x >> 5, lane = lane_id();
  const int32_t nbig = *a.big_n;
  const int64_t nwarps = (int64_t)gridDim.x * kWarps;
  for (int64_t b = blockIdx.x * (int64_t)kWarps + warp; b < nbig; b += nwarps) {
    const int64_t cell = a.big_list[b];
    Cell c;
    load_cell(a, cell, &c);
    const int32_t nfo = a.nfcell_off[cell];
    if (c.sn == 0) {  // nothing sampled here: the frontier cell carries over unchanged
      for (int32_t i = lane; i < c.fn; i += 32) {
        a.nfb_id[nfo + i] = a.fb_id[c.fo + i];
        a.nfb_pos[nfo + i] = a.fb_pos[c.fo + i];
      }
      continue;
    }
    const int32_t nb = a.nsz_prev[c.j] + a.newbase[(int64_t)c.j * a.tm.T + c.t];
    big_emit(a, c, nb, nfo, D_s[warp], N_s[warp], pD_s[warp], pN_s[warp]);
  }
}

__global__ void add_sizes_kernel(const int32_t* __restrict__ prev, const int32_t* __restrict__ add,
                                 int32_t* __restrict__ next, int32_t H, const int32_t* status) {
  if (failed(status)) return;
  for (int j = blockIdx.x * blockDim.x + threadIdx.x; j < H; j += gridDim.x * blockDim.x)
    next[j] = prev[j] + add[j];
}

}  // namespace

cudaError_t launch_dedup(const HopArgs& a, const DedupBufs& d, int num_sms, cudaStream_t st) {
  const TileMap tm{a.tile_first, a.chunk_tile, a.T};
  const int64_t ncells = (int64_t)a.T * a.H;
  int gx = (num_sms * 8 + a.H - 1) / a.H;
  if (gx < 1) gx = 1;
  const dim3 egrid(gx, a.H);
  cudaError_t e = seg_scan<int32_t, int32_t>(d.scnt, 0, d.soff, 0, nullptr, ncells, 1, ncells,
                                             true, nullptr, d.scan_scratch, a.status, st);
  if (e != cudaSuccess) return e;
  dedup_scatter_kernel<<<egrid, kThreads, 0, st>>>(d.nbr, d.ecnt, a.ecap, d.scell, d.srank,
                                                   d.soff, d.sb, a.status);
  e = cudaMemsetAsync(d.big_n, 0, sizeof(int32_t), st);
  if (e != cudaSuccess) return e;

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
  c.big_list = d.big_list;
  c.big_n = d.big_n;
  c.soff = d.soff;
  c.tile_adj_block = d.tile_adj_block;
  c.adj_flags = d.adj_flags;
  c.newcnt = d.newcnt;
  c.newbase = d.newbase;
  c.nfcnt = d.nfcnt;
  c.nfcell_off = d.nfcell_off;
  c.nfb_id = d.nfb_id;
  c.nfb_pos = d.nfb_pos;
  c.nsz_prev = d.nsz_prev;
  c.nodes = d.nodes;
  c.col = d.col;
  c.status = a.status;
  const int cgrid = num_sms * 8;
  dedup_count_kernel<<<cgrid, kThreads, 0, st>>>(c);
  dedup_count_big_kernel<<<cgrid, kThreads, 0, st>>>(c);
  e = seg_scan<int32_t, int32_t>(d.newcnt, a.T, d.newbase, a.T, nullptr, a.T, a.H, a.T, false,
                                 d.newtot, d.scan_scratch, a.status, st);
  if (e != cudaSuccess) return e;
  add_sizes_kernel<<<(a.H + 255) / 256, 256, 0, st>>>(d.nsz_prev, d.newtot, d.nsz_next, a.H,
                                                      a.status);
  e = seg_scan<int32_t, int32_t>(d.nfcnt, 0, d.nfcell_off, 0, nullptr, ncells, 1, ncells, true,
                                 nullptr, d.scan_scratch, a.status, st);
  if (e != cudaSuccess) return e;
  dedup_emit_kernel<<<cgrid, kThreads, 0, st>>>(c);
  dedup_emit_big_kernel<<<cgrid, kThreads, 0, st>>>(c);
  return cudaGetLastError();
}

}  // namespace agnes
