// common.cuh -- device helpers shared by the libagnes kernels (sm_103a).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace agnes {

// Buckets are kept per "tile": a run of consecutive node ids that lies in one
// topology block and one feature block and spans at most kTileSpan ids, so a
// tile's membership fits a 128-word bitmap.  Every multiple of kTileSpan
// starts a tile, so a node's tile is found from its 4096-id chunk plus a short
// search among the tiles that start inside that chunk.
constexpr int kTileShift = 12;
constexpr int kTileSpan = 1 << kTileShift;
constexpr int kTileWords = kTileSpan / 32;
constexpr int kWideMax = 1024;  // fanouts the warp sampler handles with its choices in shared memory

// Bits of the device status word.
enum : int32_t {
  kErrTargetRange = 1,  // a target id outside [0, N)
  kErrTargetDup = 2,    // a target repeated within a minibatch
  kErrInternal = 4,     // a capacity or consistency check failed
  kErrWaitTimeout = 8,  // a bounded wait on another CTA's progress ran out
};

struct TileMap {
  const int32_t* tile_first;  // T+1 entries, tile_first[T] = N
  const int32_t* chunk_tile;  // C+1 entries: first tile of each 4096-id chunk
  int32_t T;
};

// Tile holding node v (0 <= v < N).
__device__ __forceinline__ int32_t tile_of(const TileMap& m, int32_t v) {
  const int32_t c = v >> kTileShift;
  int32_t lo = __ldg(m.chunk_tile + c);
  int32_t hi = __ldg(m.chunk_tile + c + 1);
  while (hi - lo > 1) {
    const int32_t mid = (lo + hi) >> 1;
    if (__ldg(m.tile_first + mid) <= v)
      lo = mid;
    else
      hi = mid;
  }
  return lo;
}

// Philox4x32-10 (Salmon et al., SC'11): 10 rounds of the multiply-xor
// bijection on a 4-word counter, key bumped by the Weyl constants.
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint2 k) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r > 0) {
      k.x += 0x9E3779B9u;
      k.y += 0xBB67AE85u;
    }
    const uint32_t hi0 = __umulhi(0xD2511F53u, c.x), lo0 = 0xD2511F53u * c.x;
    const uint32_t hi1 = __umulhi(0xCD9E8D57u, c.z), lo1 = 0xCD9E8D57u * c.z;
    c = make_uint4(hi1 ^ c.y ^ k.x, lo1, hi0 ^ c.w ^ k.y, lo0);
  }
  return c;
}

__device__ __forceinline__ int lane_id() { return threadIdx.x & 31; }

// counters[idx] += 1 for every active lane, one atomic per distinct idx.
__device__ __forceinline__ void warp_agg_inc(int32_t* counters, int64_t idx, bool active) {
  const unsigned mask = __ballot_sync(0xffffffffu, active);
  if (!active) return;
  const unsigned peers = __match_any_sync(mask, (unsigned long long)idx);
  const int leader = __ffs(peers) - 1;
  if (lane_id() == leader) atomicAdd(counters + idx, __popc(peers));
}

// Takes one slot per active lane from counters[idx] by counting it down;
// returns a slot in [0, count) distinct among all takers of idx.  After every
// counted item has taken its slot the counter is back at zero.
__device__ __forceinline__ int32_t warp_agg_take(int32_t* counters, int64_t idx, unsigned mask) {
  const unsigned peers = __match_any_sync(mask, (unsigned long long)idx);
  const int leader = __ffs(peers) - 1;
  const int lane = lane_id();
  int32_t old = 0;
  if (lane == leader) old = atomicSub(counters + idx, __popc(peers));
  old = __shfl_sync(peers, old, leader);
  return old - 1 - __popc(peers & ((1u << lane) - 1u));
}

// Adds one per active lane to counters[idx] (one atomic per distinct idx) and
// returns this lane's rank among all additions to idx: the counter's value
// before it plus its rank among the warp's peers.
__device__ __forceinline__ int32_t warp_agg_add(int32_t* counters, int64_t idx, unsigned mask) {
  const unsigned peers = __match_any_sync(mask, (unsigned long long)idx);
  const int leader = __ffs(peers) - 1;
  const int lane = lane_id();
  int32_t old = 0;
  if (lane == leader) old = atomicAdd(counters + idx, __popc(peers));
  old = __shfl_sync(peers, old, leader);
  return old + __popc(peers & ((1u << lane) - 1u));
}

template <typename T>
__device__ __forceinline__ T warp_incl_scan(T x) {
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const T y = __shfl_up_sync(0xffffffffu, x, d);
    if (lane_id() >= d) x += y;
  }
  return x;
}

template <typename T>
__device__ __forceinline__ T warp_sum(T x) {
#pragma unroll
  for (int d = 16; d > 0; d >>= 1) x += __shfl_xor_sync(0xffffffffu, x, d);
  return x;
}

__device__ __forceinline__ bool failed(const int32_t* status) {
  return *(volatile const int32_t*)status != 0;
}

// Programmatic dependent launch: a kernel launched ahead of its predecessor's
// completion (a programmatic graph edge) waits here until the predecessor has
// finished and its writes are visible.  Every kernel of the hyperbatch path
// calls it first, unconditionally, so completion stays transitive along the
// chain; without a programmatic dependency it returns at once.
__device__ __forceinline__ void grid_dep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

}  // namespace agnes
