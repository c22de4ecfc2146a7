// sage.cu -- a GraphSAGE-mean layer over one sampled hop of every minibatch
// of the last hyperbatch: the consumer of the prepared blocks.  It is an
// instance of eq. (1) (Sec. 3.1): the aggregation is the mean of the
// in-neighbours' rows and the update is a fully connected layer with ReLU,
//
//   out_i = ReLU(W_self x_i + W_neigh mean_{(i,u) in hop} x_u + b).
//
// One persistent CTA per SM takes tiles of 128 dst rows of one minibatch.
// Its 16 warps aggregate the tile into shared memory as the update's input
// A = [x_dst | agg] (128 x 2 d_in, fp16, in the K-major no-swizzle layout of
// tcgen05 shared-memory operands: 8-row x 16-byte core matrices, the 16 row
// groups of a 16-byte K slice stored one after another).  One thread then
// issues the tile's chain of tcgen05.mma (M = 128, N = d_out, K = 16 each)
// against W (loaded into shared memory once per CTA, same layout) with the
// fp32 accumulator in tensor memory, and commits it to an mbarrier.  Every
// warp reads a 32-row x d_out/4 slice of the accumulator back with
// tcgen05.ld, adds the bias, applies ReLU and stores it.
//
// The aggregation reads ~(1 + deg) rows per dst row from HBM and the
// contraction is 2 * 128 * 2 d_in * d_out flops per tile, so for the sampled
// degrees the layer is bound by HBM, with the tensor cores keeping the
// update off the critical path.
#include <cuda_fp16.h>

#include <vector>

#include "../../include/agnes.h"
#include "common.cuh"
#include "internal.h"

namespace agnes {

namespace {

constexpr int kM = 128;          // dst rows per tile (the MMA's M)
constexpr int kSageThreads = 512;
constexpr int kSageWarps = kSageThreads / 32;
constexpr int kWaitIters = 1 << 24;  // mbarrier polls before giving up (~1 s)
constexpr int kIpSlots = kM + 2;     // staged indptr entries (kM + 1, padded to 16 bytes)
constexpr int kColCap = 4096;        // staged columns per tile (fanouts up to 32)
constexpr size_t kStageBytes = kIpSlots * 8 + kColCap * 4 + 16;  // + mbarrier, TMEM slot

// error word bits
constexpr int32_t kSageTimeout = 1;

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

// Byte offset of element (r, k) in a K-major no-swizzle operand of `rows`
// rows: core matrix (r / 8, k / 8) at ((k / 8) * rows / 8 + r / 8) * 128.
__device__ __forceinline__ uint32_t kmajor_off(int r, int k, int rows) {
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

struct SageArgs {
  const void* x;              // minibatch j's src rows at x + (j * x_stride + r) * d_in
  int64_t x_stride;
  const int64_t* indptr;      // minibatch j at indptr + j * indptr_stride
  int64_t indptr_stride;
  const int32_t* col;
  int64_t col_stride;
  const int32_t* tile_start;  // H + 1: first tile of each minibatch
  const int32_t* num_dst;     // host-computed per minibatch dst sizes (device copy)
  int32_t H;
  int32_t d_in, d_out;
  const __half* w;            // d_out x 2 d_in
  const float* bias;          // d_out or null
  void* out;                  // minibatch j's dst rows at out + (j * out_stride + i) * d_out
  int64_t out_stride;
  int32_t* err;
};

// 8 consecutive features of row r as fp16 (fp32 inputs are rounded).
template <typename T>
__device__ __forceinline__ uint4 load8_h(const T* row, int c);

template <>
__device__ __forceinline__ uint4 load8_h<__half>(const __half* row, int c) {
  return __ldg((const uint4*)row + c);
}

template <>
__device__ __forceinline__ uint4 load8_h<float>(const float* row, int c) {
  const float4 a = __ldg((const float4*)row + 2 * c), b = __ldg((const float4*)row + 2 * c + 1);
  uint4 r;
  __half2 h;
  h = __floats2half2_rn(a.x, a.y); r.x = *(uint32_t*)&h;
  h = __floats2half2_rn(a.z, a.w); r.y = *(uint32_t*)&h;
  h = __floats2half2_rn(b.x, b.y); r.z = *(uint32_t*)&h;
  h = __floats2half2_rn(b.z, b.w); r.w = *(uint32_t*)&h;
  return r;
}

// 8 consecutive features of a row as raw 16-byte vectors (one for fp16, two
// for fp32), loaded before they are summed so that many are in flight.
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

template <typename T, typename OutT>
__global__ void __launch_bounds__(kSageThreads, 1) sage_mean_kernel(SageArgs a) {
  extern __shared__ __align__(1024) uint8_t smem[];
  const int KT = 2 * a.d_in;        // the update's K
  const int N = a.d_out;
  uint8_t* sA = smem;                                   // kM x KT fp16
  uint8_t* sW = smem + (size_t)kM * KT * 2;             // N x KT fp16
  int64_t* s_ip = (int64_t*)(sW + (size_t)N * KT * 2);  // kM + 1 (padded to kIpSlots)
  int32_t* s_col = (int32_t*)(s_ip + kIpSlots);          // kColCap
  uint64_t* bar = (uint64_t*)(s_col + kColCap);
  uint32_t* tmem_slot = (uint32_t*)(bar + 1);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t ncols = N <= 32 ? 32 : (N <= 64 ? 64 : (N <= 128 ? 128 : 256));

  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32(tmem_slot)),
                 "r"(ncols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  if (tid == 0) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(bar)) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  // W into its K-major layout: 16-byte chunk (n, kc) = W[n][8 kc .. 8 kc + 7]
  const int kchunks = KT / 8;
  for (int q = tid; q < N * kchunks; q += kSageThreads) {
    const int n = q / kchunks, kc = q - n * kchunks;
    *(uint4*)(sW + kmajor_off(n, kc * 8, N)) = __ldg((const uint4*)(a.w + (size_t)n * KT) + kc);
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
  const uint32_t tmem = *tmem_slot;
  const uint32_t idesc = idesc_f16(kM, N);
  const uint32_t a_addr = smem_u32(sA), w_addr = smem_u32(sW);
  const int total_tiles = __ldg(a.tile_start + a.H);
  const int chunks = a.d_in / 8;  // 16-byte fp16 chunks per half of A's row
  uint32_t phase = 0;
  bool ok = true;

  for (int tile = blockIdx.x; tile < total_tiles; tile += gridDim.x) {
    int lo = 0, hi = a.H;  // minibatch of this tile: last j with tile_start[j] <= tile
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (__ldg(a.tile_start + mid) <= tile) lo = mid; else hi = mid;
    }
    const int j = lo;
    const int row0 = (tile - __ldg(a.tile_start + j)) * kM;
    const int nd = __ldg(a.num_dst + j);
    const T* x = (const T*)a.x + (size_t)j * a.x_stride * a.d_in;
    const int64_t* ip = a.indptr + (size_t)j * a.indptr_stride;
    const int32_t* cl = a.col + (size_t)j * a.col_stride;

    // stage the tile's indptr (rows past nd get empty ranges) and, when they
    // fit, its edges' columns in shared memory with coalesced loads, so the
    // row loads below do not wait on an indptr -> col chain per item
    const int rows = nd - row0 < kM ? nd - row0 : kM;
    if (tid <= kM) s_ip[tid] = __ldg(ip + row0 + (tid < rows ? tid : rows));
    __syncthreads();
    const int64_t eb = s_ip[0], ne_t = s_ip[kM] - eb;
    const bool staged = ne_t <= kColCap;
    if (staged)
      for (int64_t e = tid; e < ne_t; e += kSageThreads) s_col[e] = __ldg(cl + eb + e);
    __syncthreads();
    // aggregation: item (r, c) = row r's 8-feature chunk c; two items per
    // thread at a time, kER edges of each in flight per round
    constexpr int kER = sizeof(T) == 2 ? 8 : 4;
    for (int q0 = tid; q0 < kM * chunks; q0 += 2 * kSageThreads) {
      int r[2], c[2];
      int64_t e0[2], e1[2];
      uint4 self[2];
      float acc[2][8];
      int64_t span = 0;
#pragma unroll
      for (int k = 0; k < 2; ++k) {
        const int q = q0 + k * kSageThreads;
        r[k] = q / chunks;
        c[k] = q - r[k] * chunks;
        self[k] = make_uint4(0, 0, 0, 0);
        e0[k] = e1[k] = 0;
        if (q < kM * chunks && r[k] < rows) {
          self[k] = load8_h<T>(x + (size_t)(row0 + r[k]) * a.d_in, c[k]);
          e0[k] = s_ip[r[k]] - eb;
          e1[k] = s_ip[r[k] + 1] - eb;
        }
        span = e1[k] - e0[k] > span ? e1[k] - e0[k] : span;
#pragma unroll
        for (int f = 0; f < 8; ++f) acc[k][f] = 0.f;
      }
      for (int64_t base = 0; base < span; base += kER) {
        // indices first, then every row load, then the sums: the loads of a
        // round are independent and all in flight together
        int32_t idx[2][kER];
#pragma unroll
        for (int k = 0; k < 2; ++k)
#pragma unroll
          for (int u = 0; u < kER; ++u) {
            const int64_t e = e0[k] + base + u;
            idx[k][u] = e < e1[k] ? (staged ? s_col[e] : __ldg(cl + eb + e)) : -1;
          }
        Chunk<T> val[2][kER];
#pragma unroll
        for (int k = 0; k < 2; ++k)
#pragma unroll
          for (int u = 0; u < kER; ++u) {
            if (idx[k][u] >= 0) {
              val[k][u] = load_chunk<T>(x + (size_t)idx[k][u] * a.d_in, c[k]);
            } else {
#pragma unroll
              for (int q = 0; q < (int)(sizeof(T) / 2); ++q) val[k][u].v[q] = make_uint4(0, 0, 0, 0);
            }
          }
#pragma unroll
        for (int k = 0; k < 2; ++k)
#pragma unroll
          for (int u = 0; u < kER; ++u) add_chunk(val[k][u], acc[k]);
      }
#pragma unroll
      for (int k = 0; k < 2; ++k) {
        if (q0 + k * kSageThreads >= kM * chunks) continue;
        uint4 mean = make_uint4(0, 0, 0, 0);
        if (e1[k] > e0[k]) {
          const float deg = (float)(e1[k] - e0[k]);
          __half2 h;
          h = __floats2half2_rn(acc[k][0] / deg, acc[k][1] / deg); mean.x = *(uint32_t*)&h;
          h = __floats2half2_rn(acc[k][2] / deg, acc[k][3] / deg); mean.y = *(uint32_t*)&h;
          h = __floats2half2_rn(acc[k][4] / deg, acc[k][5] / deg); mean.z = *(uint32_t*)&h;
          h = __floats2half2_rn(acc[k][6] / deg, acc[k][7] / deg); mean.w = *(uint32_t*)&h;
        }
        *(uint4*)(sA + kmajor_off(r[k], c[k] * 8, kM)) = self[k];
        *(uint4*)(sA + kmajor_off(r[k], a.d_in + c[k] * 8, kM)) = mean;
      }
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (tid == 0) {
      asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
      // K step s covers K columns [16 s, 16 s + 16): core-matrix columns 2s, 2s+1
      for (int s = 0; s < KT / 16; ++s) {
        const uint64_t da = smem_desc(a_addr + (uint32_t)(2 * s) * (kM / 8) * 128,
                                      (kM / 8) * 128, 128);
        const uint64_t dw = smem_desc(w_addr + (uint32_t)(2 * s) * (uint32_t)(N / 8) * 128,
                                      (uint32_t)(N / 8) * 128, 128);
        mma_f16(tmem, da, dw, idesc, s > 0 ? 1u : 0u);
      }
      asm volatile(
          "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
              smem_u32(bar))
          : "memory");
    }
    const bool done = mbar_wait(smem_u32(bar), phase);
    phase ^= 1u;
    if (__syncthreads_or(!done)) {
      ok = false;
      break;
    }
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    // epilogue: warp w reads lanes 32 (w % 4) .. +31 (its rows) and the
    // column quarter w / 4, eight columns per tcgen05.ld
    {
      const int quad = warp & 3, part = warp >> 2;
      const int r = quad * 32 + lane;
      const int i = row0 + r;
      const int cols = N / 4;
      OutT* orow = (OutT*)a.out + ((size_t)j * a.out_stride + i) * N;
      for (int c0 = part * cols; c0 < (part + 1) * cols; c0 += 8) {
        uint32_t v[8];
        const uint32_t taddr = tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)c0;
        asm volatile(
            "tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
            : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]),
              "=r"(v[6]), "=r"(v[7])
            : "r"(taddr)
            : "memory");
        asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
        if (i < nd) {
          float f[8];
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            f[q] = __uint_as_float(v[q]) + (a.bias ? __ldg(a.bias + c0 + q) : 0.f);
            f[q] = f[q] > 0.f ? f[q] : 0.f;
          }
          if constexpr (sizeof(OutT) == 4) {
            ((float4*)(orow + c0))[0] = make_float4(f[0], f[1], f[2], f[3]);
            ((float4*)(orow + c0))[1] = make_float4(f[4], f[5], f[6], f[7]);
          } else {
            uint4 o;
            __half2 h;
            h = __floats2half2_rn(f[0], f[1]); o.x = *(uint32_t*)&h;
            h = __floats2half2_rn(f[2], f[3]); o.y = *(uint32_t*)&h;
            h = __floats2half2_rn(f[4], f[5]); o.z = *(uint32_t*)&h;
            h = __floats2half2_rn(f[6], f[7]); o.w = *(uint32_t*)&h;
            *(uint4*)(orow + c0) = o;
          }
        }
      }
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
  }
  if (!ok && tid == 0) atomicOr(a.err, kSageTimeout);
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
  __syncthreads();
  if (warp == 0) {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(ncols)
                 : "memory");
  }
}

size_t sage_smem_bytes(int64_t d_in, int64_t d_out) {
  return (size_t)kM * 2 * d_in * 2 + (size_t)d_out * 2 * d_in * 2 + kStageBytes;
}

bool is_device_ptr(const void* p) {
  cudaPointerAttributes attr;
  if (cudaPointerGetAttributes(&attr, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return attr.type == cudaMemoryTypeDevice || attr.type == cudaMemoryTypeManaged;
}

static_assert(kStageBytes == 17440, "the header's shared-memory formula");

// Every CTA asks for at least this much shared memory, so no two CTAs share
// an SM (and its 512 tensor-memory columns).
constexpr size_t kSageMinSmem = 120 * 1024;

template <typename T, typename OutT>
cudaError_t launch_sage(const SageArgs& a, int grid, size_t smem, cudaStream_t st) {
  if (smem < kSageMinSmem) smem = kSageMinSmem;
  cudaError_t e = cudaFuncSetAttribute(sage_mean_kernel<T, OutT>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  sage_mean_kernel<T, OutT><<<grid, kSageThreads, smem, st>>>(a);
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
  const size_t smem = sage_smem_bytes(d_in, d_out);
  if (smem > AGNES_SAGE_MAX_SMEM) {
    ctx_set_error(ctx, "d_in %lld with d_out %d needs %zu bytes of shared memory (limit %d)",
                  (long long)d_in, d_out, smem, AGNES_SAGE_MAX_SMEM);
    return AGNES_ERANGE;
  }
  if (((uintptr_t)x | (uintptr_t)w | (uintptr_t)out) % 16 != 0 ||
      ((uintptr_t)bias % 4) != 0) {
    ctx_set_error(ctx, "x, w and out must be 16-byte aligned");
    return AGNES_EINVAL;
  }
  const int H = v.H;
  int64_t max_src = 0, max_dst = 0;
  // pinned staging: error word (16 bytes), then tile_start (H + 1), num_dst (H)
  const size_t tab_bytes = sizeof(int32_t) * ((size_t)2 * H + 1);
  void* hp = nullptr;
  cudaError_t e = ctx_pinned(ctx, 16 + tab_bytes, &hp);
  if (e != cudaSuccess) {
    ctx_set_error(ctx, "agnes_sage_mean_layer: %s", cudaGetErrorString(e));
    return AGNES_ENOMEM;
  }
  int32_t* h_err = (int32_t*)hp;
  int32_t* tabs = (int32_t*)((char*)hp + 16);
  int64_t tiles = 0;
  for (int j = 0; j < H; ++j) {
    const int64_t nd = v.node_size[(size_t)hop * H + j];
    const int64_t ns = v.src_size[(size_t)hop * H + j];
    max_dst = nd > max_dst ? nd : max_dst;
    max_src = ns > max_src ? ns : max_src;
    tabs[j] = (int32_t)tiles;
    tabs[H + 1 + j] = (int32_t)nd;
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
  GraphView g;
  ctx_graph_view(ctx, &g);
  cudaStream_t st = (cudaStream_t)cuda_stream;
  void* scratch = nullptr;
  e = ctx_scratch(ctx, 16 + tab_bytes, &scratch);
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
    a.H = H;
    a.d_in = (int32_t)d_in;
    a.d_out = d_out;
    a.w = (const __half*)w;
    a.bias = bias;
    a.out = out;
    a.out_stride = out_stride_rows;
    a.err = err;
    const int grid = (int)(tiles < g.num_sms ? tiles : g.num_sms);
    if (x_dtype == AGNES_F16)
      e = out_dtype == AGNES_F32 ? launch_sage<__half, float>(a, grid, smem, st)
                                 : launch_sage<__half, __half>(a, grid, smem, st);
    else
      e = out_dtype == AGNES_F32 ? launch_sage<float, float>(a, grid, smem, st)
                                 : launch_sage<float, __half>(a, grid, smem, st);
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
    ctx_set_error(ctx, "agnes_sage_mean_layer: the tensor-core wait ran out");
    return AGNES_ETIMEOUT;
  }
  return AGNES_OK;
}
