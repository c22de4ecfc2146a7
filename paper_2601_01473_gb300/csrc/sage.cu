// sage.cu -- a GraphSAGE-mean layer over one sampled hop of every minibatch
// of the last hyperbatch: the consumer of the prepared blocks.  It is an
// instance of eq. (1) (Sec. 3.1): the aggregation is the mean of the
// in-neighbours' rows and the update is a fully connected layer with ReLU,
//
//   out_i = ReLU(W_self x_i + W_neigh mean_{(i,u) in hop} x_u + b).
//
// Two kernels.  The dst rows of minibatch j form ceil(|dst_h| / 128) tiles of
// 128 rows (the MMA's M).
//  1. sage_agg_kernel (HBM-bound gather): for every row, the mean of its
//     neighbours' rows in fp32, written with the row itself as the update's
//     input A = [x_i | mean_i] in fp16 -- each tile as the exact image of a
//     tcgen05 K-major, no-swizzle shared-memory operand (8-row x 16-byte core
//     matrices, the 16 row groups of one 16-byte K slice after one another).
//     No shared memory and no barriers, so it runs at full occupancy.
//  2. sage_gemm_kernel (persistent, warp-specialised, one CTA per SM): W is
//     loaded into shared memory once; a producer lane moves A tiles into a
//     ring of shared-memory stages with cp.async.bulk (mbarrier transaction
//     counts); an MMA lane issues each tile's tcgen05.mma chain (M = 128,
//     N = d_out, K = 16 each) into one of two TMEM accumulators; four
//     epilogue warps read the accumulator back with tcgen05.ld, add the bias,
//     apply ReLU and store -- overlapped with the next tile's copy and MMA.
// Every mbarrier wait is bounded; on timeout the kernel records an error,
// frees its tensor memory and returns.
#include <cuda_fp16.h>

#include "../../include/agnes.h"
#include "common.cuh"
#include "internal.h"

namespace agnes {

namespace {

constexpr int kM = 128;              // dst rows per tile (the MMA's M)
constexpr int kWaitIters = 1 << 24;  // mbarrier polls before giving up (~1 s)
constexpr int kAggThreads = 256;
constexpr int kGemmThreads = 256;    // warp 0 producer, warp 1 MMA, warps 4-7 epilogue
constexpr int kBarBytes = 128;       // mbarriers + TMEM address slot
// Every GEMM CTA asks for at least this much shared memory, so no two CTAs
// share an SM (and its 512 tensor-memory columns).
constexpr size_t kSageMinSmem = 120 * 1024;

constexpr int32_t kSageTimeout = 1;  // error word bits

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

// Byte offset of element (r, k) in a K-major no-swizzle operand of `rows`
// rows: core matrix (r / 8, k / 8) at ((k / 8) * rows / 8 + r / 8) * 128.
__host__ __device__ __forceinline__ uint32_t kmajor_off(int r, int k, int rows) {
  return (uint32_t)((((k >> 3) * (rows >> 3)) + (r >> 3)) * 128 + (r & 7) * 16 + (k & 7) * 2);
}

// tcgen05 shared-memory matrix descriptor, no swizzle: start address, the
// byte distance between core matrices adjacent in K (leading) and in M/N
// (stride), and the fixed version bits 46-48 = 0b001.
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr, uint32_t lbo, uint32_t sbo) {
  return (uint64_t)((addr & 0x3FFFF) >> 4) | ((uint64_t)((lbo & 0x3FFFF) >> 4) << 16) |
         ((uint64_t)((sbo & 0x3FFFF) >> 4) << 32) | (1ull << 46);
}

// Instruction descriptor of kind::f16: fp32 accumulator (bits 4-5 = 1), fp16
// A and B (bits 7-9, 10-12 = 0), both K-major (bits 15, 16 = 0), N >> 3 at
// bits 17-22, M >> 4 at bits 24-28.
__device__ __forceinline__ uint32_t idesc_f16(int m, int n) {
  return (1u << 4) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(m >> 4) << 24);
}

__device__ __forceinline__ void mma_f16(uint32_t tmem_d, uint64_t a, uint64_t b, uint32_t idesc,
                                        uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}"
      :
      : "r"(tmem_d), "l"(a), "l"(b), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void mma_commit(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
      : "memory");
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void mbar_arrive_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}

// Waits for the phase with the given parity to complete; false after
// kWaitIters polls.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
  for (int it = 0; it < kWaitIters; ++it) {
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(bar), "r"(parity)
        : "memory");
    if (done) return true;
    if (it >= 32) __nanosleep(64);
  }
  return false;
}

// Bulk copy of `bytes` (a multiple of 16, both addresses 16-byte aligned)
// from global memory into shared memory, completing a transaction on bar.
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes,
                                         uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
          "r"(dst),
      "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}

// 8 consecutive features of a row as raw 16-byte vectors (one for fp16, two
// for fp32).
template <typename T>
struct Chunk {
  uint4 v[sizeof(T) / 2];
};

template <typename T>
__device__ __forceinline__ Chunk<T> load_chunk(const T* row, int c) {
  Chunk<T> ch;
#pragma unroll
  for (int q = 0; q < (int)(sizeof(T) / 2); ++q)
    ch.v[q] = __ldg((const uint4*)row + (sizeof(T) / 2) * c + q);
  return ch;
}

__device__ __forceinline__ void add_chunk(const Chunk<__half>& ch, float* acc) {
  const __half2* h = (const __half2*)&ch.v[0];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const float2 f = __half22float2(h[q]);
    acc[2 * q] += f.x;
    acc[2 * q + 1] += f.y;
  }
}

__device__ __forceinline__ void add_chunk(const Chunk<float>& ch, float* acc) {
  const float* f = (const float*)&ch.v[0];
#pragma unroll
  for (int q = 0; q < 8; ++q) acc[q] += f[q];
}

__device__ __forceinline__ uint4 to_half8(const float* f) {
  uint4 o;
  __half2 h;
  h = __floats2half2_rn(f[0], f[1]); o.x = *(uint32_t*)&h;
  h = __floats2half2_rn(f[2], f[3]); o.y = *(uint32_t*)&h;
  h = __floats2half2_rn(f[4], f[5]); o.z = *(uint32_t*)&h;
  h = __floats2half2_rn(f[6], f[7]); o.w = *(uint32_t*)&h;
  return o;
}

struct SageArgs {
  const void* x;              // minibatch j's src rows at x + (j * x_stride + r) * d_in
  int64_t x_stride;
  const int64_t* indptr;      // minibatch j at indptr + j * indptr_stride
  int64_t indptr_stride;
  const int32_t* col;
  int64_t col_stride;
  const int32_t* tile_start;  // H + 1: first tile of each minibatch
  const int32_t* num_dst;     // H: |dst_h| per minibatch
  const int32_t* tile_mb;     // per tile: its minibatch
  int32_t H;
  int32_t d_in, d_out;
  uint8_t* A;                 // tiles x (kM x 2 d_in fp16), each tile a shared-memory image
  const __half* w;            // d_out x 2 d_in
  const float* bias;          // d_out or null
  void* out;                  // minibatch j's dst rows at out + (j * out_stride + i) * d_out
  int64_t out_stride;
  int32_t stages;             // A stages in the GEMM's shared memory
  int32_t* err;
};


// Items (R, c): row R of the tile space, 8-feature chunk c of x; each
// thread takes kAggU items kAggThreads apart at a time, every load stage
// issued for all of them before the next.  Writes the chunk of x_i and of
// mean_i into the row's A tile (zeros past |dst_h|).
constexpr int kAggU = 1;

template <typename T>
__global__ void __launch_bounds__(kAggThreads, 5) sage_agg_kernel(SageArgs a, int64_t rows_total) {
  constexpr int kER = sizeof(T) == 2 ? 8 : 4;  // edges in flight per item and round
  constexpr int U = kAggU;
  const int chunks = a.d_in / 8;
  const int64_t items = rows_total * chunks;
  const size_t tile_bytes = (size_t)kM * 2 * a.d_in * 2;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t q0 = blockIdx.x * (int64_t)blockDim.x * U + threadIdx.x; q0 < items;
       q0 += stride * U) {
    int c[U], tile[U], r[U];
    bool row_ok[U];
    const T* x[U];
    const int32_t* cl[U];
    int64_t e0[U], e1[U], span = 0;
    Chunk<T> sc[U];
#pragma unroll
    for (int k = 0; k < U; ++k) {
      const int64_t q = q0 + (int64_t)k * blockDim.x;
      const int64_t R = q < items ? q / chunks : 0;
      c[k] = (int)(q - R * chunks);
      tile[k] = (int)(R / kM);
      r[k] = (int)(R - (int64_t)tile[k] * kM);
      row_ok[k] = false;
      e0[k] = e1[k] = 0;
      if (q < items) {
        const int j = __ldg(a.tile_mb + tile[k]);
        const int i = (tile[k] - __ldg(a.tile_start + j)) * kM + r[k];
        if (i < __ldg(a.num_dst + j)) {
          row_ok[k] = true;
          x[k] = (const T*)a.x + (size_t)j * a.x_stride * a.d_in;
          cl[k] = a.col + (size_t)j * a.col_stride;
          const int64_t* ip = a.indptr + (size_t)j * a.indptr_stride;
          sc[k] = load_chunk<T>(x[k] + (size_t)i * a.d_in, c[k]);
          e0[k] = __ldg(ip + i);
          e1[k] = __ldg(ip + i + 1);
          span = e1[k] - e0[k] > span ? e1[k] - e0[k] : span;
        }
      }
    }
    float acc[U][8];
#pragma unroll
    for (int k = 0; k < U; ++k)
#pragma unroll
      for (int z = 0; z < 8; ++z) acc[k][z] = 0.f;
    for (int64_t base = 0; base < span; base += kER) {
      int32_t idx[U][kER];
#pragma unroll
      for (int k = 0; k < U; ++k)
#pragma unroll
        for (int u = 0; u < kER; ++u)
          idx[k][u] = e0[k] + base + u < e1[k] ? __ldg(cl[k] + e0[k] + base + u) : -1;
      Chunk<T> val[U][kER];
#pragma unroll
      for (int k = 0; k < U; ++k)
#pragma unroll
        for (int u = 0; u < kER; ++u) {
          if (idx[k][u] >= 0) {
            val[k][u] = load_chunk<T>(x[k] + (size_t)idx[k][u] * a.d_in, c[k]);
          } else {
#pragma unroll
            for (int z = 0; z < (int)(sizeof(T) / 2); ++z)
              val[k][u].v[z] = make_uint4(0, 0, 0, 0);
          }
        }
#pragma unroll
      for (int k = 0; k < U; ++k)
#pragma unroll
        for (int u = 0; u < kER; ++u) add_chunk(val[k][u], acc[k]);
    }
#pragma unroll
    for (int k = 0; k < U; ++k) {
      const int64_t q = q0 + (int64_t)k * blockDim.x;
      if (q >= items) continue;
      uint4 self = make_uint4(0, 0, 0, 0), mean = make_uint4(0, 0, 0, 0);
      if (row_ok[k]) {
        if constexpr (sizeof(T) == 2) {
          self = sc[k].v[0];
        } else {
          const float* f = (const float*)&sc[k].v[0];
          float g[8];
#pragma unroll
          for (int z = 0; z < 8; ++z) g[z] = f[z];
          self = to_half8(g);
        }
        if (e1[k] > e0[k]) {
          const float deg = (float)(e1[k] - e0[k]);
#pragma unroll
          for (int z = 0; z < 8; ++z) acc[k][z] /= deg;
          mean = to_half8(acc[k]);
        }
      }
      uint8_t* At = a.A + (size_t)tile[k] * tile_bytes;
      *(uint4*)(At + kmajor_off(r[k], c[k] * 8, kM)) = self;
      *(uint4*)(At + kmajor_off(r[k], a.d_in + c[k] * 8, kM)) = mean;
    }
  }
}

template <typename OutT>
__global__ void __launch_bounds__(kGemmThreads, 1) sage_gemm_kernel(SageArgs a) {
  extern __shared__ __align__(1024) uint8_t smem[];
  const int KT = 2 * a.d_in;
  const int N = a.d_out;
  const int S = a.stages;
  const uint32_t tile_bytes = (uint32_t)kM * KT * 2;
  uint8_t* sW = smem;                                 // N x KT fp16
  uint8_t* sA = smem + (size_t)N * KT * 2;            // S stages of kM x KT fp16
  uint64_t* bars = (uint64_t*)(sA + (size_t)S * tile_bytes);
  // full[0..S), empty[4..4+S), dfull[8..10), dempty[10..12), then the TMEM slot
  const uint32_t bar0 = smem_u32(bars);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t ncols = 2 * N <= 64 ? 64 : (2 * N <= 128 ? 128 : (2 * N <= 256 ? 256 : 512));
  uint32_t* tmem_slot = (uint32_t*)(bars + 12);
#define AGNES_FULL(s) (bar0 + 8u * (uint32_t)(s))
#define AGNES_EMPTY(s) (bar0 + 8u * (uint32_t)(4 + (s)))
#define AGNES_DFULL(d) (bar0 + 8u * (uint32_t)(8 + (d)))
#define AGNES_DEMPTY(d) (bar0 + 8u * (uint32_t)(10 + (d)))

  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_slot)),
                 "r"(ncols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(AGNES_FULL(s), 1);
      mbar_init(AGNES_EMPTY(s), 1);
    }
    for (int d = 0; d < 2; ++d) {
      mbar_init(AGNES_DFULL(d), 1);
      mbar_init(AGNES_DEMPTY(d), 4);  // one arrival per epilogue warp
    }
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  // W into its K-major layout: 16-byte chunk (n, kc) = W[n][8 kc .. 8 kc + 7]
  const int kchunks = KT / 8;
  for (int q = tid; q < N * kchunks; q += kGemmThreads) {
    const int n = q / kchunks, kc = q - n * kchunks;
    *(uint4*)(sW + kmajor_off(n, kc * 8, N)) = __ldg((const uint4*)(a.w + (size_t)n * KT) + kc);
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *tmem_slot;
  const int total_tiles = __ldg(a.tile_start + a.H);
  bool ok = true;

  if (warp == 0) {
    // producer: A tile k of this CTA into stage k % S
    if (lane == 0) {
      int k = 0;
      for (int tile = blockIdx.x; tile < total_tiles; tile += gridDim.x, ++k) {
        const int s = k % S;
        if (k >= S && !mbar_wait(AGNES_EMPTY(s), (uint32_t)((k / S - 1) & 1))) {
          ok = false;
          break;
        }
        mbar_arrive_tx(AGNES_FULL(s), tile_bytes);
        bulk_g2s(smem_u32(sA + (size_t)s * tile_bytes), a.A + (size_t)tile * tile_bytes,
                 tile_bytes, AGNES_FULL(s));
      }
    }
  } else if (warp == 1) {
    // MMA issuer: tile k from stage k % S into accumulator k % 2
    if (lane == 0) {
      const uint32_t idesc = idesc_f16(kM, N);
      const uint32_t w_addr = smem_u32(sW);
      int k = 0;
      for (int tile = blockIdx.x; tile < total_tiles; tile += gridDim.x, ++k) {
        const int s = k % S, d = k & 1;
        if (!mbar_wait(AGNES_FULL(s), (uint32_t)((k / S) & 1)) ||
            (k >= 2 && !mbar_wait(AGNES_DEMPTY(d), (uint32_t)((k / 2 - 1) & 1)))) {
          ok = false;
          break;
        }
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        const uint32_t a_addr = smem_u32(sA + (size_t)s * tile_bytes);
        const uint32_t dcol = tmem + (uint32_t)(d * N);
        // K step t covers K columns [16 t, 16 t + 16): core-matrix columns 2t, 2t+1
        for (int t = 0; t < KT / 16; ++t) {
          const uint64_t da = smem_desc(a_addr + (uint32_t)(2 * t) * (kM / 8) * 128,
                                        (kM / 8) * 128, 128);
          const uint64_t dw = smem_desc(w_addr + (uint32_t)(2 * t) * (uint32_t)(N / 8) * 128,
                                        (uint32_t)(N / 8) * 128, 128);
          mma_f16(dcol, da, dw, idesc, t > 0 ? 1u : 0u);
        }
        mma_commit(AGNES_EMPTY(s));  // the stage is free once these MMAs have read it
        mma_commit(AGNES_DFULL(d));  // and the accumulator is complete
      }
    }
  } else if (warp >= 4) {
    // epilogue: warp w reads TMEM lanes 32 (w % 4) .. +31 (its rows)
    const int quad = warp & 3;
    int k = 0;
    for (int tile = blockIdx.x; tile < total_tiles; tile += gridDim.x, ++k) {
      const int d = k & 1;
      if (!mbar_wait(AGNES_DFULL(d), (uint32_t)((k / 2) & 1))) {
        ok = false;
        break;
      }
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      const int j = __ldg(a.tile_mb + tile);
      const int i = (tile - __ldg(a.tile_start + j)) * kM + quad * 32 + lane;
      const bool valid = i < __ldg(a.num_dst + j);
      OutT* orow = (OutT*)a.out + ((size_t)j * a.out_stride + i) * N;
      for (int c0 = 0; c0 < N; c0 += 32) {  // 32 columns per tcgen05.ld, one wait
        uint32_t v[32];
        const uint32_t taddr = tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)(d * N + c0);
        asm volatile(
            "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, "
            "%10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, "
            "%26, %27, %28, %29, %30, %31}, [%32];"
            : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]),
              "=r"(v[6]), "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]),
              "=r"(v[12]), "=r"(v[13]), "=r"(v[14]), "=r"(v[15]), "=r"(v[16]), "=r"(v[17]),
              "=r"(v[18]), "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]),
              "=r"(v[24]), "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]),
              "=r"(v[30]), "=r"(v[31])
            : "r"(taddr)
            : "memory");
        asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
        if (valid) {
#pragma unroll
          for (int g = 0; g < 4; ++g) {
            float f[8];
#pragma unroll
            for (int q = 0; q < 8; ++q) {
              const int cc = c0 + 8 * g + q;
              f[q] = __uint_as_float(v[8 * g + q]) + (a.bias ? __ldg(a.bias + cc) : 0.f);
              f[q] = f[q] > 0.f ? f[q] : 0.f;
            }
            if constexpr (sizeof(OutT) == 4) {
              ((float4*)(orow + c0 + 8 * g))[0] = make_float4(f[0], f[1], f[2], f[3]);
              ((float4*)(orow + c0 + 8 * g))[1] = make_float4(f[4], f[5], f[6], f[7]);
            } else {
              *(uint4*)(orow + c0 + 8 * g) = to_half8(f);
            }
          }
        }
      }
      asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
      __syncwarp();
      if (lane == 0) mbar_arrive(AGNES_DEMPTY(d));
    }
  }
#undef AGNES_FULL
#undef AGNES_EMPTY
#undef AGNES_DFULL
#undef AGNES_DEMPTY
  if (!ok) atomicOr(a.err, kSageTimeout);
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (warp == 0) {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(ncols)
                 : "memory");
  }
}

// Shared memory of the GEMM kernel with `stages` A stages.
size_t gemm_smem_bytes(int64_t d_in, int64_t d_out, int stages) {
  return (size_t)d_out * 2 * d_in * 2 + (size_t)stages * kM * 2 * d_in * 2 + kBarBytes;
}

bool is_device_ptr(const void* p) {
  cudaPointerAttributes attr;
  if (cudaPointerGetAttributes(&attr, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return attr.type == cudaMemoryTypeDevice || attr.type == cudaMemoryTypeManaged;
}

template <typename T, typename OutT>
cudaError_t launch_sage(const SageArgs& a, int64_t tiles, int num_sms, cudaStream_t st) {
  const int64_t rows = tiles * kM;
  const int64_t items = rows * (a.d_in / 8);
  int64_t agg_grid = resident_grid((const void*)sage_agg_kernel<T>, kAggThreads, num_sms);
  const int64_t per_cta = (int64_t)kAggThreads * kAggU;
  if (agg_grid * per_cta > items) agg_grid = (items + per_cta - 1) / per_cta;
  sage_agg_kernel<T><<<(unsigned)agg_grid, kAggThreads, 0, st>>>(a, rows);
  size_t smem = gemm_smem_bytes(a.d_in, a.d_out, a.stages);
  if (smem < kSageMinSmem) smem = kSageMinSmem;
  cudaError_t e = cudaFuncSetAttribute(sage_gemm_kernel<OutT>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const int grid = (int)(tiles < num_sms ? tiles : num_sms);
  sage_gemm_kernel<OutT><<<grid, kGemmThreads, smem, st>>>(a);
  return cudaGetLastError();
}

}  // namespace

}  // namespace agnes

using namespace agnes;

extern "C" agnes_status agnes_sage_mean_layer(agnes_ctx* ctx, int32_t hop, const void* x,
                                              int32_t x_dtype, int64_t x_stride_rows,
                                              int64_t d_in, const void* w, const float* bias,
                                              int32_t d_out, void* out, int32_t out_dtype,
                                              int64_t out_stride_rows, void* cuda_stream) {
  if (!ctx || !x || !w || !out) {
    ctx_set_error(ctx, "ctx, x, w and out must be non-NULL");
    return AGNES_EINVAL;
  }
  GraphView g;
  ctx_graph_view(ctx, &g);
  DeviceGuard dg(g.device);
  if (!dg.ok()) {
    ctx_set_error(ctx, "cudaSetDevice(%d) failed", g.device);
    return AGNES_ECUDA;
  }
  agnes_hyperbatch_view v;
  agnes_status rc = agnes_fetch_hyperbatch(ctx, &v);
  if (rc != AGNES_OK) return rc;
  if (hop < 0 || hop >= v.K) {
    ctx_set_error(ctx, "hop %d outside [0, %d)", hop, v.K);
    return AGNES_EINVAL;
  }
  if ((x_dtype != AGNES_F32 && x_dtype != AGNES_F16) ||
      (out_dtype != AGNES_F32 && out_dtype != AGNES_F16)) {
    ctx_set_error(ctx, "x_dtype and out_dtype must be AGNES_F32 or AGNES_F16");
    return AGNES_EINVAL;
  }
  if (d_in < 8 || d_in % 8 != 0 || d_out < 32 || d_out > 256 || d_out % 32 != 0) {
    ctx_set_error(ctx, "d_in must be a positive multiple of 8 and d_out a multiple of 32 in "
                       "[32, 256]");
    return AGNES_EINVAL;
  }
  int stages = 2;
  if (gemm_smem_bytes(d_in, d_out, stages) > AGNES_SAGE_MAX_SMEM) stages = 1;
  if (gemm_smem_bytes(d_in, d_out, stages) > AGNES_SAGE_MAX_SMEM) {
    ctx_set_error(ctx, "d_in %lld with d_out %d needs %zu bytes of shared memory (limit %d)",
                  (long long)d_in, d_out, gemm_smem_bytes(d_in, d_out, 1), AGNES_SAGE_MAX_SMEM);
    return AGNES_ERANGE;
  }
  if (((uintptr_t)x | (uintptr_t)w | (uintptr_t)out) % 16 != 0 ||
      ((uintptr_t)bias % 4) != 0) {
    ctx_set_error(ctx, "x, w and out must be 16-byte aligned");
    return AGNES_EINVAL;
  }
  const int H = v.H;
  int64_t max_src = 0, max_dst = 0;
  // pinned staging: error word (16 bytes), then tile_start (H + 1), num_dst
  // (H), tile_mb (one per tile)
  int64_t tiles = 0;
  for (int j = 0; j < H; ++j) tiles += ((int64_t)v.node_size[(size_t)hop * H + j] + kM - 1) / kM;
  const size_t tab_bytes = sizeof(int32_t) * ((size_t)2 * H + 1 + (size_t)tiles);
  void* hp = nullptr;
  cudaError_t e = ctx_pinned(ctx, 16 + tab_bytes, &hp);
  if (e != cudaSuccess) {
    ctx_set_error(ctx, "agnes_sage_mean_layer: %s", cudaGetErrorString(e));
    return AGNES_ENOMEM;
  }
  int32_t* h_err = (int32_t*)hp;
  int32_t* tabs = (int32_t*)((char*)hp + 16);
  tiles = 0;
  for (int j = 0; j < H; ++j) {
    const int64_t nd = v.node_size[(size_t)hop * H + j];
    const int64_t ns = v.src_size[(size_t)hop * H + j];
    max_dst = nd > max_dst ? nd : max_dst;
    max_src = ns > max_src ? ns : max_src;
    tabs[j] = (int32_t)tiles;
    tabs[H + 1 + j] = (int32_t)nd;
    for (int64_t t = tiles; t < tiles + (nd + kM - 1) / kM; ++t) tabs[2 * H + 1 + t] = j;
    tiles += (nd + kM - 1) / kM;
  }
  tabs[H] = (int32_t)tiles;
  if (x_stride_rows < max_src || out_stride_rows < max_dst) {
    ctx_set_error(ctx, "x_stride_rows must be >= %lld and out_stride_rows >= %lld",
                  (long long)max_src, (long long)max_dst);
    return AGNES_EINVAL;
  }
  if (!is_device_ptr(x) || !is_device_ptr(w) || !is_device_ptr(out) ||
      (bias && !is_device_ptr(bias))) {
    ctx_set_error(ctx, "x, w, bias and out must be device memory");
    return AGNES_EINVAL;
  }
  cudaStream_t st = (cudaStream_t)cuda_stream;
  // device scratch: error word and tables, then (256-byte aligned) the A tiles
  const size_t a_off = (16 + tab_bytes + 255) & ~(size_t)255;
  const size_t a_bytes = (size_t)tiles * kM * 2 * (size_t)d_in * 2;
  void* scratch = nullptr;
  e = ctx_scratch(ctx, a_off + a_bytes, &scratch);
  int32_t* err = (int32_t*)scratch;
  int32_t* d_tabs = (int32_t*)((char*)scratch + 16);
  if (e == cudaSuccess) e = cudaMemsetAsync(err, 0, sizeof(int32_t), st);
  if (e == cudaSuccess) e = cudaMemcpyAsync(d_tabs, tabs, tab_bytes, cudaMemcpyHostToDevice, st);
  if (e == cudaSuccess && tiles > 0) {
    SageArgs a;
    a.x = x;
    a.x_stride = x_stride_rows;
    a.indptr = v.indptr[hop];
    a.indptr_stride = v.indptr_stride[hop];
    a.col = v.col[hop];
    a.col_stride = v.col_stride[hop];
    a.tile_start = d_tabs;
    a.num_dst = d_tabs + H + 1;
    a.tile_mb = d_tabs + 2 * H + 1;
    a.H = H;
    a.d_in = (int32_t)d_in;
    a.d_out = d_out;
    a.A = (uint8_t*)scratch + a_off;
    a.w = (const __half*)w;
    a.bias = bias;
    a.out = out;
    a.out_stride = out_stride_rows;
    a.stages = stages;
    a.err = err;
    if (x_dtype == AGNES_F16)
      e = out_dtype == AGNES_F32 ? launch_sage<__half, float>(a, tiles, g.num_sms, st)
                                 : launch_sage<__half, __half>(a, tiles, g.num_sms, st);
    else
      e = out_dtype == AGNES_F32 ? launch_sage<float, float>(a, tiles, g.num_sms, st)
                                 : launch_sage<float, __half>(a, tiles, g.num_sms, st);
  }
  *h_err = 0;
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(h_err, err, sizeof(int32_t), cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) {
    ctx_set_error(ctx, "agnes_sage_mean_layer: %s", cudaGetErrorString(e));
    return e == cudaErrorMemoryAllocation ? AGNES_ENOMEM : AGNES_ECUDA;
  }
  if (*h_err & kSageTimeout) {
    ctx_set_error(ctx, "agnes_sage_mean_layer: a tensor-core or copy wait ran out");
    return AGNES_ETIMEOUT;
  }
  return AGNES_OK;
}
