// sample.cu -- bucketing of the targets and per-hop neighbour sampling.
//
// Bucket matrix (Sec. 3.4 (3), Algorithm 1's Bck_{i,j}): frontier entries are
// kept per (tile, minibatch) cell in tile-major, minibatch-minor order, sorted
// by node id inside a cell, each with its global output row
// g = j * capK + position.  A topology block's requests are therefore one
// contiguous run of the bucket, and sampling walks the bucket in order, so the
// block is read once for all minibatches of the hyperbatch (Sec. 3.3) and its
// adjacency data is reused out of L2.
//
// Sampling (Sec. 3.1, Algorithm 1's Sample): up to k neighbours per frontier
// node, uniformly without replacement; all of them in CSR order when
// deg <= k, else Floyd's algorithm (Bentley & Floyd, CACM 1987) with
// Philox4x32-10 draws keyed on (seed; v, hop, slot, g).  For k <= 32 a group
// of k lanes handles one frontier node (32 / k nodes per warp round): lane s
// draws slot s's candidate in parallel and the k-step collision resolution
// runs over warp shuffles.  Above 32 a warp takes 32 slots at a time,
// checking each candidate against the earlier chunks' choices (in shared
// memory up to kWideMax, in a hash set in global memory beyond).  The count
// kernel's (first edge, degree) per frontier entry lets the fill read them
// coalesced.
#include "common.cuh"
#include "internal.h"

namespace agnes {

namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;

// ---- bucketing of the targets ------------------------------------------------

__global__ void __launch_bounds__(kThreads)
targets_count_kernel(const int32_t* __restrict__ nodes, int64_t capK, int32_t H, int32_t B,
                     int32_t N, TileMap tm, int32_t* __restrict__ fcnt, int32_t* status) {
  grid_dep_wait();
  const int64_t total = (int64_t)H * B;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i0 = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) & ~31ll; i0 < total;
       i0 += stride) {
    const int64_t i = i0 + lane_id();
    bool active = i < total;
    int64_t cell = 0;
    if (active) {
      const int32_t j = (int32_t)(i / B);
      const int32_t v = nodes[j * capK + (i - (int64_t)j * B)];
      if (v < 0 || v >= N) {
        atomicOr(status, kErrTargetRange);
        active = false;
      } else {
        cell = (int64_t)tile_of(tm, v) * H + j;
      }
    }
    warp_agg_inc(fcnt, cell, active);
  }
}

__global__ void __launch_bounds__(kThreads)
targets_scatter_kernel(const int32_t* __restrict__ nodes, int64_t capK, int32_t H, int32_t B,
                       int32_t N, TileMap tm, int32_t* __restrict__ fcnt,
                       const int32_t* __restrict__ fcell_off, int32_t* __restrict__ tmp_id,
                       int32_t* __restrict__ tmp_pos, const int32_t* status) {
  grid_dep_wait();
  if (failed(status)) return;
  const int64_t total = (int64_t)H * B;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i0 = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) & ~31ll; i0 < total;
       i0 += stride) {
    const int64_t i = i0 + lane_id();
    bool active = i < total;
    int32_t v = 0, j = 0;
    int64_t cell = 0;
    if (active) {
      j = (int32_t)(i / B);
      v = nodes[j * capK + (i - (int64_t)j * B)];
      active = v >= 0 && v < N;
      if (active) cell = (int64_t)tile_of(tm, v) * H + j;
    }
    const unsigned mask = __ballot_sync(0xffffffffu, active);
    if (active) {
      const int32_t slot = fcell_off[cell] + warp_agg_take(fcnt, cell, mask);
      tmp_id[slot] = v;
      tmp_pos[slot] = (int32_t)(j * capK + (i - (int64_t)j * B));
    }
  }
}

// Orders each cell's targets by id and flags a target repeated within a
// minibatch.  A warp scans 32 consecutive cells and skips empty ones; a cell
// of at most 32 targets is ranked in registers (each lane counts the smaller
// ids), a bigger one by popcount ranks in a bitmap over its tile.
__global__ void __launch_bounds__(kThreads)
targets_sort_kernel(const int32_t* __restrict__ fcell_off, int64_t ncells, int32_t H, TileMap tm,
                    const int32_t* __restrict__ tmp_id, const int32_t* __restrict__ tmp_pos,
                    int32_t* __restrict__ fb_id, int32_t* __restrict__ fb_pos, int32_t* status) {
  grid_dep_wait();
  if (failed(status)) return;
  __shared__ uint32_t bits_s[kWarps][kTileWords];
  __shared__ int32_t pref_s[kWarps][kTileWords];
  const int warp = threadIdx.x >> 5, lane = lane_id();
  uint32_t* bits = bits_s[warp];
  int32_t* pref = pref_s[warp];
  const int64_t nchunks = (ncells + 31) / 32;
  const int64_t nwarps = (int64_t)gridDim.x * kWarps;
  for (int64_t ch = blockIdx.x * (int64_t)kWarps + warp; ch < nchunks; ch += nwarps) {
    const int64_t my_cell = ch * 32 + lane;
    int32_t my_o = 0, my_n = 0;
    if (my_cell < ncells) {
      my_o = fcell_off[my_cell];
      my_n = fcell_off[my_cell + 1] - my_o;
    }
    unsigned todo = __ballot_sync(0xffffffffu, my_n > 0);
    while (todo) {
      const int k = __ffs(todo) - 1;
      todo &= todo - 1u;
      const int32_t o = __shfl_sync(0xffffffffu, my_o, k);
      const int32_t n = __shfl_sync(0xffffffffu, my_n, k);
      if (n <= 32) {
        const bool act = lane < n;
        const int32_t v = act ? tmp_id[o + lane] : 0x7fffffff;
        const int32_t p = act ? tmp_pos[o + lane] : 0;
        const unsigned amask = n >= 32 ? 0xffffffffu : ((1u << n) - 1u);
        const unsigned peers = __match_any_sync(0xffffffffu, v);  // every lane takes part
        if (act && __popc(peers & amask) > 1) atomicOr(status, kErrTargetDup);
        int32_t r = 0;
        for (int q = 0; q < n; ++q) r += __shfl_sync(0xffffffffu, v, q) < v;
        if (act) {
          fb_id[o + r] = v;
          fb_pos[o + r] = p;
        }
        continue;
      }
      const int32_t t = (int32_t)((ch * 32 + k) / H);
      const int32_t base = tm.tile_first[t];
      const int32_t words = (tm.tile_first[t + 1] - base + 31) >> 5;
      for (int w = lane; w < words; w += 32) bits[w] = 0;
      __syncwarp();
      for (int32_t i = lane; i < n; i += 32) {
        const int32_t lu = tmp_id[o + i] - base;
        const uint32_t bit = 1u << (lu & 31);
        if (atomicOr(&bits[lu >> 5], bit) & bit) atomicOr(status, kErrTargetDup);
      }
      __syncwarp();
      int32_t c[4], sum = 0;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int w = lane * 4 + q;
        c[q] = w < words ? __popc(bits[w]) : 0;
        sum += c[q];
      }
      int32_t run = warp_incl_scan(sum) - sum;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        pref[lane * 4 + q] = run;
        run += c[q];
      }
      __syncwarp();
      for (int32_t i = lane; i < n; i += 32) {
        const int32_t v = tmp_id[o + i];
        const int32_t lu = v - base;
        const int32_t w = lu >> 5;
        const int32_t r = pref[w] + __popc(bits[w] & ((1u << (lu & 31)) - 1u));
        fb_id[o + r] = v;
        fb_pos[o + r] = tmp_pos[o + i];
      }
      __syncwarp();
    }
  }
}

// ---- sampling --------------------------------------------------------------------

// Per frontier entry i (bucket order): the node's count of sampled edges
// min(deg, k) at its minibatch position (for the edge offsets' scan), and
// (first edge, degree) in fbd[i] for the fill, which then reads them
// coalesced instead of the offsets at random.
template <typename OffT>
__global__ void __launch_bounds__(kThreads)
sample_count_kernel(const int32_t* __restrict__ fb_id, const int32_t* __restrict__ fb_pos,
                    const int32_t* total_ptr, const OffT* __restrict__ off, int64_t capK,
                    int64_t cap_prev, int32_t k, int32_t* __restrict__ cnt,
                    longlong2* __restrict__ fbd, const int32_t* status) {
  grid_dep_wait();
  if (failed(status)) return;
  const int64_t total = *total_ptr;
  const uint32_t capk32 = (uint32_t)capK;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int32_t v = fb_id[i];
    const uint32_t g = (uint32_t)fb_pos[i];
    const uint32_t j = g / capk32;
    const uint32_t pos = g - j * capk32;
    const int64_t base = (int64_t)__ldg(off + v);
    const int64_t d = (int64_t)__ldg(off + v + 1) - base;
    cnt[j * cap_prev + pos] = (int32_t)(d < k ? d : k);
    fbd[i] = make_longlong2(base, d);
  }
}

struct FillArgs {
  TileMap tm;
  // frontier entries [fcell_off[cell_lo], fcell_off[cell_hi]) are sampled
  const int32_t* fcell_off;
  int64_t cell_lo, cell_hi;
  // streamed topology: edge lists of resident physical blocks in the graph
  // buffer (slot * epb edges each); blk_slot[b] < 0 means not resident
  const int32_t* tile_adj_block;
  const int32_t* blk_slot;
  const int64_t* blk_e0;
  const int32_t* gbuf;
  int64_t epb, hdr, bb;
  int32_t H;
  int32_t* scnt;   // T*H per-cell counters of sampled ids (zero on entry)
  int32_t* scell;  // per edge: its (tile, minibatch) cell
  int32_t* srank;  // per edge: its rank within the cell
  const int32_t* fb_id;
  const int32_t* fb_pos;
  const longlong2* fbd;  // per frontier entry: (first edge, degree) of its node
  const int64_t* indptr;
  const int32_t* indices;
  int32_t* nbr;
  int64_t capK, cap_prev, ecap;
  int32_t k, hop;
  const uint64_t* key;  // device: {seed, first minibatch id}
  int32_t* status;
  bool packed;        // record rank << 12 | tile-local id in nbr, no srank (the dedup's
                      // sampled bucket is packed)
  int32_t* hset;      // fanouts above kWideMax: per-warp hash sets of chosen positions
  int32_t hset_log2;  // each of 2^hset_log2 entries
};

// The sampling key, read from device memory once per thread, so that one
// captured launch sequence serves every seed and minibatch id.
struct Key {
  uint32_t lo, hi;
  uint64_t gid0;
};

__device__ __forceinline__ Key load_key(const uint64_t* key) {
  const uint64_t seed = __ldg(key);
  return Key{(uint32_t)seed, (uint32_t)(seed >> 32), __ldg(key + 1)};
}

// Where the sampler reads neighbour entries.
enum EdgeSrc : int {
  kEdgesInPlace = 0,  // a.indices (HBM, or the device view of pinned host memory)
  kEdgesBuffer = 1,   // the graph buffer: every needed block is resident
  kEdgesCached = 2,   // the topology cache where the block is cached, else in place
};

// Neighbour at position pos of node v (edges off_v .. off_v + deg).  In the
// graph buffer or the topology cache the edge sits in the slot of its
// physical block: v's first block, plus, for an object larger than a block,
// the block its byte offset (after the header) falls in.
template <int kSrc>
__device__ __forceinline__ int32_t edge_at(const FillArgs& a, int32_t v, int64_t off_v,
                                           int64_t deg, int64_t pos) {
  if (kSrc == kEdgesInPlace) return __ldg(a.indices + off_v + pos);
  int64_t b = __ldg(a.tile_adj_block + tile_of(a.tm, v));
  if (a.hdr + 4 * deg > a.bb) b += (a.hdr + 4 * pos) / a.bb;
  const int32_t slot = __ldg(a.blk_slot + b);
  if (slot < 0) {
    if (kSrc == kEdgesCached) return __ldg(a.indices + off_v + pos);
    atomicOr(a.status, kErrInternal);  // cannot happen: the host made every needed block resident
    return 0;
  }
  return __ldg(a.gbuf + (int64_t)slot * a.epb + (off_v + pos - __ldg(a.blk_e0 + b)));
}

__device__ __forceinline__ int64_t draw(const FillArgs& a, const Key& key, int32_t v, int32_t s,
                                        uint64_t gid, int64_t J) {
  const uint4 x = philox4x32_10(
      make_uint4((uint32_t)v, ((uint32_t)a.hop << 24) | (uint32_t)s, (uint32_t)gid,
                 (uint32_t)(gid >> 32)),
      make_uint2(key.lo, key.hi));
  const uint64_t r = ((uint64_t)x.y << 32) | (uint64_t)x.x;
  return (int64_t)__umul64hi(r, (uint64_t)(J + 1));
}

// Records sampled edge e = (j, eidx) with neighbour u: its id, its
// (tile, minibatch) cell and its rank within the cell (one atomic per distinct
// cell of the warp), so the bucketing scatter after the scan needs no atomics.
// Called by all 32 lanes; lanes without an edge pass has = false.  Cell
// indices fit 31 bits (T * H < 2^31).
__device__ __forceinline__ void emit_edges(const FillArgs& a, bool has, int32_t u, uint32_t j,
                                           int64_t eidx) {
  const int32_t t = tile_of(a.tm, has ? u : 0);
  const uint32_t cell = (uint32_t)t * (uint32_t)a.H + j;
  // the id, or with a packed sampled bucket its tile-local id
  const int32_t val = a.packed ? u - __ldg(a.tm.tile_first + t) : u;
  const unsigned peers = __match_any_sync(0xffffffffu, has ? cell : 0xffffffffu);
  const int lane = lane_id();
  const int leader = __ffs(peers) - 1;
  int32_t old = 0;
  if (has && lane == leader) old = atomicAdd(a.scnt + cell, __popc(peers));
  old = __shfl_sync(0xffffffffu, old, leader);
  if (has) {
    const int64_t at = (int64_t)j * a.ecap + eidx;
    const int32_t rank = old + __popc(peers & ((1u << lane) - 1u));
    a.scell[at] = (int32_t)cell;
    if (a.packed) {  // rank < ecap <= 2^20 beside the 12-bit tile-local id
      a.nbr[at] = (rank << 12) | val;
    } else {
      a.nbr[at] = val;
      a.srank[at] = rank;
    }
  }
}

// k <= 32: k lanes per frontier node (lane s draws slot s), 32 / k nodes per
// warp round; the lanes past them (32 mod k) idle.  The round runs without
// divergent branches: every lane draws (a node of degree <= k takes its
// first d edges instead) and the collision shuffles span the whole warp.
template <int kSrc>
__global__ void __launch_bounds__(kThreads, 8) sample_fill_kernel(FillArgs a) {
  grid_dep_wait();
  if (failed(a.status)) return;
  const Key key = load_key(a.key);
  const int64_t E0 = a.fcell_off[a.cell_lo], E1 = a.fcell_off[a.cell_hi];
  const int k = a.k;
  const int groups = 32 / k;
  const int lane = lane_id();
  const int sub = lane / k, s = lane - sub * k;
  const int g0 = sub * k;  // the group's first lane (>= 32 - k for idle lanes)
  const bool member = sub < groups;
  const uint32_t capk32 = (uint32_t)a.capK;
  const int64_t warp0 = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t e0 = E0 + warp0 * groups; e0 < E1; e0 += nwarps * groups) {
    const int64_t i = e0 + sub;
    const bool live = member && i < E1;
    int32_t v = 0;
    uint32_t g = 0;
    longlong2 bd = make_longlong2(0, 0);
    if (live) {
      v = a.fb_id[i];
      g = (uint32_t)a.fb_pos[i];
      bd = a.fbd[i];
    }
    const int64_t base = bd.x, d = bd.y;
    const uint32_t j = g / capk32;
    const uint32_t pos = g - j * capk32;
    int64_t eidx = s;
    if (live) eidx += a.indptr[j * (a.cap_prev + 1) + pos];
    // Floyd's algorithm: slot s draws t in [0, J], J = d - k + s, and takes J
    // when an earlier slot of the node holds t
    const int64_t J = d - k + s;
    const int64_t t = draw(a, key, v, s, key.gid0 + j, J);
    bool collided = false;
    if (__any_sync(0xffffffffu, d > (int64_t)0xffffffffu)) {  // positions past 32 bits
      for (int q = 0; q < k; ++q) {
        const int64_t cq = __shfl_sync(0xffffffffu, collided ? J : t, g0 + q);
        if (s > q && t == cq) collided = true;
      }
    } else {
      const uint32_t t32 = (uint32_t)t, J32 = (uint32_t)J;
      for (int q = 0; q < k; ++q) {
        const uint32_t cq = __shfl_sync(0xffffffffu, collided ? J32 : t32, g0 + q);
        if (s > q && t32 == cq) collided = true;
      }
    }
    const bool small = d <= k;
    const bool has = live && (!small || s < d);
    int32_t u = 0;
    if (has) u = edge_at<kSrc>(a, v, base, d, small ? (int64_t)s : collided ? J : t);
    emit_edges(a, has, u, j, eidx);
  }
}

// One warp per frontier node for fanouts above 32: slots are drawn 32 at a
// time; each candidate is checked against the choices of earlier chunks (kept
// in shared memory) and then resolved within its chunk by shuffles.
template <int kSrc>
__global__ void __launch_bounds__(kThreads) sample_fill_wide_kernel(FillArgs a) {
  grid_dep_wait();
  if (failed(a.status)) return;
  __shared__ int32_t chosen_s[kWarps][kWideMax];
  const int warp = threadIdx.x >> 5, lane = lane_id();
  int32_t* chosen = chosen_s[warp];
  const Key key = load_key(a.key);
  const int64_t E0 = a.fcell_off[a.cell_lo], E1 = a.fcell_off[a.cell_hi];
  const uint32_t capk32 = (uint32_t)a.capK;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t i = E0 + ((blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5); i < E1;
       i += nwarps) {
    const int32_t v = a.fb_id[i];
    const uint32_t g = (uint32_t)a.fb_pos[i];
    const uint32_t j = g / capk32;
    const uint32_t pos = g - j * capk32;
    const longlong2 bd = a.fbd[i];
    const int64_t base = bd.x, d = bd.y;
    const int64_t ebase = a.indptr[j * (a.cap_prev + 1) + pos];
    if (d <= a.k) {
      for (int64_t q0 = 0; q0 < d; q0 += 32) {
        const int64_t q = q0 + lane;
        const bool has = q < d;
        emit_edges(a, has, has ? edge_at<kSrc>(a, v, base, d, q) : 0, j, ebase + q);
      }
      continue;
    }
    for (int c0 = 0; c0 < a.k; c0 += 32) {
      const int s = c0 + lane;
      const bool valid = s < a.k;
      const int64_t J = d - a.k + s;
      const int64_t t = valid ? draw(a, key, v, s, key.gid0 + j, J) : -1;
      bool collided = false;
      for (int q = 0; q < c0; ++q) collided |= (chosen[q] == t);
      const int m = min(32, a.k - c0);
      for (int q = 0; q < m; ++q) {
        const int64_t mine = collided ? J : t;
        const int64_t cq = __shfl_sync(0xffffffffu, mine, q);
        if (lane > q && t == cq) collided = true;
      }
      const int64_t c = collided ? J : t;
      if (valid) chosen[s] = (int32_t)c;
      emit_edges(a, valid, valid ? edge_at<kSrc>(a, v, base, d, c) : 0, j, ebase + s);
      __syncwarp();
    }
  }
}

// ---- fanouts above kWideMax -----------------------------------------------------
//
// One warp per frontier node, slots drawn 32 at a time as in the wide sampler;
// the positions chosen by earlier chunks live in the warp's own open-addressing
// hash set in global memory (2^hset_log2 >= 2k entries, so it is at most half
// full and every probe sequence ends at an empty entry within the table),
// cleared for each node.  Lookups bypass L1 (__ldcg): the set's entries are
// written by the warp's atomics at L2.
constexpr int32_t kHsetEmpty = -1;

__device__ __forceinline__ uint32_t hset_slot(int32_t key, uint32_t mask) {
  return ((uint32_t)key * 0x9E3779B1u) & mask;  // Fibonacci hashing, low bits
}

__device__ __forceinline__ bool hset_contains(const int32_t* T, uint32_t mask, int32_t key) {
  uint32_t h = hset_slot(key, mask);
  for (uint32_t probe = 0; probe <= mask; ++probe) {
    const int32_t v = __ldcg(T + h);
    if (v == key) return true;
    if (v == kHsetEmpty) return false;
    h = (h + 1u) & mask;
  }
  return false;
}

// Inserts key (distinct from the keys other lanes insert at the same time).
__device__ __forceinline__ void hset_insert(int32_t* T, uint32_t mask, int32_t key) {
  uint32_t h = hset_slot(key, mask);
  for (uint32_t probe = 0; probe <= mask; ++probe) {
    const int32_t old = atomicCAS(T + h, kHsetEmpty, key);
    if (old == kHsetEmpty || old == key) return;
    h = (h + 1u) & mask;
  }
}

template <int kSrc>
__global__ void __launch_bounds__(kThreads) sample_fill_huge_kernel(FillArgs a) {
  grid_dep_wait();
  if (failed(a.status)) return;
  const int lane = lane_id();
  const Key key = load_key(a.key);
  const int64_t E0 = a.fcell_off[a.cell_lo], E1 = a.fcell_off[a.cell_hi];
  const uint32_t capk32 = (uint32_t)a.capK;
  const int64_t gw = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const uint32_t mask = (1u << a.hset_log2) - 1u;
  int32_t* T = a.hset + (gw << a.hset_log2);
  for (int64_t i = E0 + gw; i < E1; i += nwarps) {
    const int32_t v = a.fb_id[i];
    const uint32_t g = (uint32_t)a.fb_pos[i];
    const uint32_t j = g / capk32;
    const uint32_t pos = g - j * capk32;
    const longlong2 bd = a.fbd[i];
    const int64_t base = bd.x, d = bd.y;
    const int64_t ebase = a.indptr[j * (a.cap_prev + 1) + pos];
    if (d <= a.k) {
      for (int64_t q0 = 0; q0 < d; q0 += 32) {
        const int64_t q = q0 + lane;
        const bool has = q < d;
        emit_edges(a, has, has ? edge_at<kSrc>(a, v, base, d, q) : 0, j, ebase + q);
      }
      continue;
    }
    for (uint32_t w = (uint32_t)lane; w <= (mask >> 2); w += 32)
      reinterpret_cast<int4*>(T)[w] = make_int4(kHsetEmpty, kHsetEmpty, kHsetEmpty, kHsetEmpty);
    __syncwarp();
    for (int c0 = 0; c0 < a.k; c0 += 32) {
      const int s = c0 + lane;
      const bool valid = s < a.k;
      const int64_t J = d - a.k + s;
      const int64_t t = valid ? draw(a, key, v, s, key.gid0 + j, J) : -1;
      bool collided = valid && hset_contains(T, mask, (int32_t)t);
      const int m = min(32, a.k - c0);
      for (int q = 0; q < m; ++q) {
        const int64_t mine = collided ? J : t;
        const int64_t cq = __shfl_sync(0xffffffffu, mine, q);
        if (lane > q && t == cq) collided = true;
      }
      const int64_t c = collided ? J : t;
      if (valid) hset_insert(T, mask, (int32_t)c);
      emit_edges(a, valid, valid ? edge_at<kSrc>(a, v, base, d, c) : 0, j, ebase + s);
      __syncwarp();  // the chunk's inserts are seen by the next chunk's lookups
    }
    __syncwarp();  // every lookup of this node is done before the next clear
  }
}

}  // namespace

int64_t huge_fanout_tables(int32_t k, int num_sms, int32_t* log2, int32_t* grid) {
  *log2 = 0;
  *grid = 0;
  if (k <= kWideMax) return 0;
  int32_t l = 2;
  while ((1 << l) < 2 * k) ++l;
  int g = resident_grid((const void*)sample_fill_huge_kernel<kEdgesInPlace>, kThreads, num_sms);
  const int64_t budget_entries = (int64_t)1 << 28;  // 1 GiB of tables at most
  const int64_t max_warps = budget_entries >> l;
  if ((int64_t)g * kWarps > max_warps) g = (int)(max_warps / kWarps);
  if (g < 1) g = 1;
  *log2 = l;
  *grid = g;
  return ((int64_t)g * kWarps) << l;
}

cudaError_t launch_bucket_targets(int32_t* nodes, int64_t capK, int32_t H, int32_t B, int32_t N,
                                  const int32_t* tile_first, const int32_t* chunk_tile, int32_t T,
                                  int32_t* fcnt, int32_t* fcell_off, int32_t* tmp_id,
                                  int32_t* tmp_pos, int32_t* fb_id, int32_t* fb_pos,
                                  int64_t* scan_scratch, uint64_t* flat_scratch, int32_t* status,
                                  int num_sms, cudaStream_t st) {
  const TileMap tm{tile_first, chunk_tile, T};
  const int64_t ncells = (int64_t)T * H;
  const int grid = resident_grid((const void*)targets_count_kernel, kThreads, num_sms);
  targets_count_kernel<<<grid, kThreads, 0, st>>>(nodes, capK, H, B, N, tm, fcnt, status);
  cudaError_t e = cells_scan(fcnt, fcell_off, ncells, flat_scratch, scan_scratch, status, st);
  if (e != cudaSuccess) return e;
  targets_scatter_kernel<<<resident_grid((const void*)targets_scatter_kernel, kThreads, num_sms),
                           kThreads, 0, st>>>(nodes, capK, H, B, N, tm, fcnt, fcell_off,
                                                    tmp_id, tmp_pos, status);
  targets_sort_kernel<<<resident_grid((const void*)targets_sort_kernel, kThreads, num_sms),
                        kThreads, 0, st>>>(fcell_off, ncells, H, tm, tmp_id, tmp_pos,
                                                 fb_id, fb_pos, status);
  return cudaGetLastError();
}

static __global__ void set_key_kernel(uint64_t* key, uint64_t seed, uint64_t first_gid) {
  grid_dep_wait();
  key[0] = seed;
  key[1] = first_gid;
}

cudaError_t launch_set_key(uint64_t* key, uint64_t seed, uint64_t first_gid, cudaStream_t st) {
  set_key_kernel<<<1, 1, 0, st>>>(key, seed, first_gid);
  return cudaGetLastError();
}

cudaError_t launch_sample_count(const HopArgs& a, const int32_t* fb_id, const int32_t* fb_pos,
                                const int32_t* fcell_off, int32_t* cnt, int num_sms,
                                cudaStream_t st) {
  const int32_t* total = fcell_off + (int64_t)a.T * a.H;
  if (a.offsets_bits == 32)
    sample_count_kernel<int32_t><<<resident_grid((const void*)sample_count_kernel<int32_t>,
                                                 kThreads, num_sms),
                                   kThreads, 0, st>>>(
        fb_id, fb_pos, total, (const int32_t*)a.offsets, a.capK, a.cap_prev, a.k, cnt,
        reinterpret_cast<longlong2*>(a.fbd), a.status);
  else
    sample_count_kernel<int64_t><<<resident_grid((const void*)sample_count_kernel<int64_t>,
                                                 kThreads, num_sms),
                                   kThreads, 0, st>>>(
        fb_id, fb_pos, total, (const int64_t*)a.offsets, a.capK, a.cap_prev, a.k, cnt,
        reinterpret_cast<longlong2*>(a.fbd), a.status);
  return cudaGetLastError();
}

template <int kSrc>
static void launch_fill_typed(const FillArgs& f, int k, int huge_grid, int num_sms,
                              cudaStream_t st) {
  if (k <= 32)
    sample_fill_kernel<kSrc><<<resident_grid((const void*)sample_fill_kernel<kSrc>, kThreads,
                                             num_sms),
                               kThreads, 0, st>>>(f);
  else if (k <= kWideMax)
    sample_fill_wide_kernel<kSrc><<<resident_grid((const void*)sample_fill_wide_kernel<kSrc>,
                                                  kThreads, num_sms),
                                    kThreads, 0, st>>>(f);
  else
    sample_fill_huge_kernel<kSrc><<<huge_grid, kThreads, 0, st>>>(f);
}

cudaError_t launch_sample_fill(const HopArgs& a, const int32_t* fb_id, const int32_t* fb_pos,
                               const int32_t* fcell_off, const int64_t* indptr, int32_t* nbr,
                               int32_t* scnt, int32_t* scell, int32_t* srank,
                               const FillRange& r, int num_sms, cudaStream_t st) {
  FillArgs f;
  f.tm = TileMap{a.tile_first, a.chunk_tile, a.T};
  f.fcell_off = fcell_off;
  f.cell_lo = r.cell_lo;
  f.cell_hi = r.cell_hi;
  f.tile_adj_block = r.tile_adj_block;
  f.blk_slot = r.blk_slot;
  f.blk_e0 = r.blk_e0;
  f.gbuf = r.gbuf;
  f.epb = r.epb;
  f.hdr = a.offsets_bits / 8;
  f.bb = r.bb;
  f.H = a.H;
  f.scnt = scnt;
  f.scell = scell;
  f.srank = srank;
  f.fb_id = fb_id;
  f.fb_pos = fb_pos;
  f.fbd = reinterpret_cast<const longlong2*>(a.fbd);
  f.indptr = indptr;
  f.indices = a.indices;
  f.nbr = nbr;
  f.capK = a.capK;
  f.cap_prev = a.cap_prev;
  f.ecap = a.ecap;
  f.k = a.k;
  f.hop = a.hop;
  f.key = a.key;
  f.status = a.status;
  f.hset = a.hset;
  f.hset_log2 = a.hset_log2;
  f.packed = a.sb_packed;
  if (a.k > kWideMax && (a.hset == nullptr || a.hset_grid < 1)) return cudaErrorInvalidValue;
  const int src = r.gbuf == nullptr ? kEdgesInPlace : r.in_place_fallback ? kEdgesCached
                                                                            : kEdgesBuffer;
  if (src == kEdgesInPlace)
    launch_fill_typed<kEdgesInPlace>(f, a.k, a.hset_grid, num_sms, st);
  else if (src == kEdgesBuffer)
    launch_fill_typed<kEdgesBuffer>(f, a.k, a.hset_grid, num_sms, st);
  else
    launch_fill_typed<kEdgesCached>(f, a.k, a.hset_grid, num_sms, st);
  return cudaGetLastError();
}

}  // namespace agnes
