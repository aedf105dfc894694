// K1 encode: l = E(x), one hidden layer (Sec. 3.2.1):
//   h = ReLU(s (W1 x) + b1),  l = W2 h + b2.
//
// Tensor-core version (tcgen05, sm_103a), persistent and warp-specialised:
// one CTA per SM keeps W1 and W2 in shared memory and walks 128-row tiles (the
// 128 TMEM lanes of its accumulators). Layer 1 runs in chunks of 128 hidden
// units: one thread issues tcgen05.mma (kind::f16, fp16 operands, fp32
// accumulation in TMEM) over the X tile and the chunk of W1; eight epilogue
// warps read each accumulator back with tcgen05.ld, apply scale, bias and
// ReLU, and write the chunk as fp16 pairs back into TMEM with tcgen05.st,
// where it is the A operand of the layer-2 MMAs that accumulate
// l [128 x N2] (N2 = b padded to 16 or 32) against W2. Two layer-1
// accumulators, two hidden chunks and two layer-2 accumulators let the tensor
// pipe work on the next chunk while the epilogue converts the previous one;
// four converter warps turn the next X tile into fp16 meanwhile (two
// buffers where shared memory allows; uint8 inputs are exact in fp16; the
// input scale is applied to the fp32 accumulator). A tile's logits are
// stored after the next tile's first chunk, when its layer-2 MMAs are done.
// Every hand-off is an mbarrier (tcgen05.commit, or thread arrivals). Shared
// memory operands sit in the canonical K-major no-swizzle layout
// (nr_tc_kmajor_off), in which the host stores W1 and W2.
//
// Every hand-off wait is bounded (1 s, or the limit nr_params.wait_limit_us
// sets); when one expires every role stops, the CTA waits for its MMAs in
// flight (bounded by 1 s whatever the limit), records NR_DEV_TIMEOUT, frees
// its TMEM and returns.
//
// Encoders with hidden layers after the first run layer by layer on a second
// tensor-core kernel (encode_layer_kernel). What neither takes (shapes
// outside their limits, input rows not 16-byte aligned) runs on the
// CUDA-core kernels at the end of the file.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>
#include <string.h>

#include "nr_internal.cuh"

namespace {

// ------------------------------------------------------------ tcgen05 helpers
__device__ __forceinline__ uint32_t smem_u32(const void *p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;\n" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t phase) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(bar), "r"(phase)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;\n" : "=l"(t));
  return t;
}
// wait for the barrier's phase to complete, for at most ~1 s
__device__ __forceinline__ bool mbar_wait_bounded(uint32_t bar, uint32_t phase) {
  const uint64_t t0 = global_ns();
  while (!mbar_try_wait(bar, phase))
    if (global_ns() - t0 > 1000000000ull) return false;
  return true;
}
__device__ __forceinline__ void tc_alloc(uint32_t slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(slot),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tc_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::: "memory");
}
__device__ __forceinline__ void tc_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(taddr), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory");
}
__device__ __forceinline__ void fence_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
}
__device__ __forceinline__ void tc_mma_f16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                           uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void tc_commit(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(bar)
      : "memory");
}
__device__ __forceinline__ void tc_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,"
      "%24,%25,%26,%27,%28,%29,%30,%31}, [%32];\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
}
__device__ __forceinline__ void tc_wait_ld() {
  asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory");
}

// shared-memory matrix descriptor: start, leading (K) and stride (8-row group)
// byte offsets, descriptor version 1, no swizzle
__device__ __forceinline__ uint64_t smem_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  return (uint64_t)((saddr >> 4) & 0x3FFFu) | ((uint64_t)((lbo >> 4) & 0x3FFFu) << 16) |
         ((uint64_t)((sbo >> 4) & 0x3FFFu) << 32) | (1ull << 46);
}
// instruction descriptor, kind::f16: D fp32, A and B fp16, both K-major
__host__ __device__ constexpr uint32_t mma_idesc(int M, int N) {
  return (1u << 4) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

// ------------------------------------------------------------ tensor-core kernel
constexpr int kRows = 128;     // rows per tile = TMEM lanes of the accumulators
constexpr int kHC = 128;       // hidden units per layer-1 chunk
constexpr int kEpiWarps = 8;   // two per TMEM lane group, one column half of a chunk each
constexpr int kConvWarps = 4;
constexpr int kWarpMma = 0, kWarpEpi = 1, kWarpConv = kWarpEpi + kEpiWarps;
constexpr int kTcThreads = 32 * (kWarpConv + kConvWarps);  // 416
constexpr int kEpiThreads = 32 * kEpiWarps, kConvThreads = 32 * kConvWarps;
// TMEM columns: layer-1 accumulators at 0 and 128, layer-2 accumulators at 256
// and 288, the hidden chunk as the fp16 A operand of layer 2 (two values a
// column) at 320 and 384
constexpr uint32_t kTmemCols = 512, kTmemAcc2 = 256, kTmemHid = 320;

struct TcBars {
  uint64_t xfull[2], xempty[2];    // X tiles: converters -> MMA -> converters
  uint64_t a1full[2], a1empty[2];  // layer-1 accumulators: MMA -> epilogue -> MMA
  uint64_t hfull[2], hempty[2];    // hidden chunks in TMEM: epilogue -> MMA -> epilogue
  uint64_t a2full[2], a2empty[2];  // layer-2 accumulators
  uint64_t drain;                  // every MMA of the CTA complete
  uint32_t tmem_slot;
  int abort;                       // a wait expired: every role stops
};

// byte offsets of the shared-memory regions for a shape with nxb X buffers
struct TcLayout {
  uint32_t x, w1, w2, b1, b2, bars, total;
};
__host__ __device__ inline TcLayout tc_layout(int D, int H, int n2, int nxb) {
  TcLayout L;
  uint32_t o = 0;
  L.x = o;  o += (uint32_t)nxb * kRows * (uint32_t)D * 2u;  // fp16 X tiles
  L.w1 = o; o += (uint32_t)H * (uint32_t)D * 2u;            // all of W1, resident
  L.w2 = o; o += (uint32_t)n2 * (uint32_t)H * 2u;           // all of W2, resident
  L.b1 = o; o += (uint32_t)H * 4u;
  L.b2 = o; o += 32u * 4u;
  L.bars = o; o += (uint32_t)sizeof(TcBars);
  L.total = o;
  return L;
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("{\n .reg .b64 st;\n mbarrier.arrive.shared::cta.b64 st, [%0];\n}\n" ::"r"(bar)
               : "memory");
}
// layer-2 MMA with A read from TMEM (a_tmem: its first column), B from shared memory
__device__ __forceinline__ void tc_mma_f16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc,
                                              uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n}\n" ::"r"(d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void tc_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}
__device__ __forceinline__ void tc_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,"
      "%25,%26,%27,%28,%29,%30,%31,%32};\n" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),
      "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]),
      "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]),
      "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}
__device__ __forceinline__ void tc_wait_st() {
  asm volatile("tcgen05.wait::st.sync.aligned;\n" ::: "memory");
}
__device__ __forceinline__ bool mbar_test_wait(uint32_t bar, uint32_t phase) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(bar), "r"(phase)
      : "memory");
  return ok != 0;
}
// Waits for the barrier phase of the given parity. Gives up when another role
// has given up, or after wait_ns nanoseconds, which makes every role give up;
// wait_ns < 0: gives up unless the phase is complete when first tested.
__device__ __forceinline__ bool wait_or_abort(uint32_t bar, uint32_t parity, volatile int *abort,
                                              int64_t wait_ns) {
  if (wait_ns < 0) {
    if (mbar_test_wait(bar, parity)) return true;
    *abort = 1;
    return false;
  }
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  for (;;) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*abort) return false;
    if (global_ns() - t0 > (uint64_t)wait_ns) {
      *abort = 1;
      return false;
    }
  }
}
// the same, one decision for the whole warp (all lanes wait)
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int *abort,
                                          int64_t wait_ns) {
  return __all_sync(0xffffffffu, wait_or_abort(bar, parity, abort, wait_ns)) != 0;
}
// 16 bytes of uint8 as 16 fp16 values, exactly: 0x64XX is the fp16 number 1024 + XX
__device__ __forceinline__ void u8x16_to_f16(const uint4 v, uint4 &lo, uint4 &hi) {
  const __half2 k1024 = __halves2half2(__ushort_as_half(0x6400), __ushort_as_half(0x6400));
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  uint32_t o[8];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint32_t p0 = __byte_perm(w[i], 0x64646464u, 0x4140), p1 = __byte_perm(w[i], 0x64646464u, 0x4342);
    const __half2 h0 = __hsub2(*reinterpret_cast<const __half2 *>(&p0), k1024);
    const __half2 h1 = __hsub2(*reinterpret_cast<const __half2 *>(&p1), k1024);
    o[2 * i] = *reinterpret_cast<const uint32_t *>(&h0);
    o[2 * i + 1] = *reinterpret_cast<const uint32_t *>(&h1);
  }
  lo = make_uint4(o[0], o[1], o[2], o[3]);
  hi = make_uint4(o[4], o[5], o[6], o[7]);
}

// The converter warps' role in the tensor-core encoders: each X tile of 128
// rows -> fp16 operand in the K-major core-matrix layout of buffer tile % nxb
// (xempty: the buffer is free; xfull: it is written, kConvThreads arrivals).
// ct: the thread's index among the converter threads.
template <int DT>
__device__ __forceinline__ void tc_convert_tiles(const void *__restrict__ x, int D, int kx, int nxb,
                                                 int64_t nq, int64_t ntiles, uint32_t x_bytes,
                                                 unsigned char *smem_x, uint64_t *xfull,
                                                 uint64_t *xempty, volatile int *abort,
                                                 int64_t wait_ns, int ct) {
  // eight consecutive threads cover eight rows of one 16-byte K chunk, so a
  // warp's stores fill whole 128-byte core matrices
  // item j of this thread: row rr of the tile and piece pc of the row (16 source
  // bytes = 2 K chunks for uint8, one K chunk of 8 floats for fp32), the same
  // for every tile; k / per by a 16-bit reciprocal, exact for k < 256, per <= 16
  const int per = DT == 0 ? D / 16 : kx;  // pieces per row = items per thread (<= 8, <= 16)
  const uint32_t inv = (65536u + (uint32_t)per - 1u) / (uint32_t)per;
  auto item = [&](int j, int &rr, int &pc) {
    const uint32_t k = (uint32_t)(ct >> 3) + 16u * (uint32_t)j, q = (k * inv) >> 16;
    pc = (int)(k - q * (uint32_t)per);
    rr = (int)q * 8 + (ct & 7);
  };
  uint32_t it = 0;
  for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x, ++it) {
    const int xb = nxb == 2 ? (int)(it & 1) : 0;
    const uint32_t xpar = ((nxb == 2 ? it >> 1 : it) & 1u) ^ 1u;  // previous use of the buffer
    unsigned char *sX = smem_x + (size_t)xb * x_bytes;
    const int64_t row0 = tile * kRows;
    const int rows = nq - row0 < kRows ? (int)(nq - row0) : kRows;  // rows of this tile
    bool ok = true;
    if (DT == 0) {
      const uint8_t *xs = static_cast<const uint8_t *>(x) + row0 * D;
      uint4 v[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        int rr, pc;
        item(j, rr, pc);
        v[j] = make_uint4(0u, 0u, 0u, 0u);
        if (j < per && rr < rows) v[j] = __ldg(reinterpret_cast<const uint4 *>(xs + rr * D + pc * 16));
      }
      ok = warp_wait(smem_u32(&xempty[xb]), xpar, abort, wait_ns);
      if (ok) {
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          if (j >= per) break;
          int rr, pc;
          item(j, rr, pc);
          uint4 lo, hi;
          u8x16_to_f16(v[j], lo, hi);
          *reinterpret_cast<uint4 *>(sX + nr_tc_kmajor_off(rr, 2 * pc, kx)) = lo;
          *reinterpret_cast<uint4 *>(sX + nr_tc_kmajor_off(rr, 2 * pc + 1, kx)) = hi;
        }
      }
    } else {
      const float *xs = static_cast<const float *>(x) + row0 * D;
#pragma unroll
      for (int j0 = 0; j0 < 16; j0 += 8) {
        if (j0 >= per || !ok) break;
        float4 u[8], w[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          int rr, pc;
          item(j0 + j, rr, pc);
          u[j] = w[j] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
          if (j0 + j < per && rr < rows) {
            const float4 *s4 = reinterpret_cast<const float4 *>(xs + rr * D + pc * 8);
            u[j] = __ldg(s4);
            w[j] = __ldg(s4 + 1);
          }
        }
        if (j0 == 0) ok = warp_wait(smem_u32(&xempty[xb]), xpar, abort, wait_ns);
        if (!ok) break;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          if (j0 + j >= per) break;
          int rr, pc;
          item(j0 + j, rr, pc);
          const __half2 h0 = __floats2half2_rn(u[j].x, u[j].y), h1 = __floats2half2_rn(u[j].z, u[j].w);
          const __half2 h2 = __floats2half2_rn(w[j].x, w[j].y), h3 = __floats2half2_rn(w[j].z, w[j].w);
          *reinterpret_cast<uint4 *>(sX + nr_tc_kmajor_off(rr, pc, kx)) =
              make_uint4(*reinterpret_cast<const uint32_t *>(&h0), *reinterpret_cast<const uint32_t *>(&h1),
                         *reinterpret_cast<const uint32_t *>(&h2), *reinterpret_cast<const uint32_t *>(&h3));
        }
      }
    }
    if (!ok) break;
    fence_async_smem();
    mbar_arrive(smem_u32(&xfull[xb]));
  }
}

// Persistent, warp-specialised: each CTA (one per SM) keeps W1 and W2 in
// shared memory and takes 128-row tiles tile = blockIdx.x, + gridDim.x, ...:
//   converter warps  X tile -> fp16 operand (nxb = 2 buffers, or 1 for wide shapes)
//   MMA thread       layer 1 of chunk g (128 hidden units) into accumulator g % 2,
//                    then layer 2 of chunk g - 1 with its A operand in TMEM
//   epilogue warps   accumulator -> ReLU(s acc + b1) -> fp16 hidden chunk in TMEM
//                    (buffer g % 2); after the next tile's first chunk, the
//                    tile's layer-2 accumulator + b2 -> out (float4 stores if
//                    vec_out: b % 4 == 0 and out 16-byte aligned)
// so that the tensor pipe runs layer 1 of the next chunk while the epilogue
// turns the previous one into the layer-2 operand.
template <int DT>
__global__ void __launch_bounds__(kTcThreads, 1)
    encode_tc_kernel(const void *__restrict__ x, int D, int H, int b, int n2, int nxb, int vec_out,
                     float s,
                     const __half *__restrict__ W1p, const float *__restrict__ b1,
                     const __half *__restrict__ W2p, const float *__restrict__ b2, int64_t nq,
                     float *__restrict__ out, int *err, int64_t wait_ns) {
  extern __shared__ __align__(1024) unsigned char smem[];
  const TcLayout L = tc_layout(D, H, n2, nxb);
  TcBars &B = *reinterpret_cast<TcBars *>(smem + L.bars);
  volatile int *abort = &B.abort;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int kx = D / 8;      // 16-byte K chunks per row of X and W1
  const int nc = H / kHC;    // layer-1 chunks per tile
  const uint32_t x_bytes = (uint32_t)kRows * D * 2, w1_bytes = (uint32_t)kHC * D * 2;
  const uint32_t w2_bytes = (uint32_t)n2 * kHC * 2;  // one chunk of W2
  const int64_t ntiles = (nq + kRows - 1) / kRows;
  const uint32_t sbase = smem_u32(smem);
  float *sb1 = reinterpret_cast<float *>(smem + L.b1);
  float *sb2 = reinterpret_cast<float *>(smem + L.b2);

  if (warp == kWarpMma) {
    tc_alloc(smem_u32(&B.tmem_slot), kTmemCols);
    tc_relinquish();
  }
  if (tid == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&B.xfull[i]), kConvThreads);
      mbar_init(smem_u32(&B.xempty[i]), 1);
      mbar_init(smem_u32(&B.a1full[i]), 1);
      mbar_init(smem_u32(&B.a1empty[i]), kEpiThreads);
      mbar_init(smem_u32(&B.hfull[i]), kEpiThreads);
      mbar_init(smem_u32(&B.hempty[i]), 1);
      mbar_init(smem_u32(&B.a2full[i]), 1);
      mbar_init(smem_u32(&B.a2empty[i]), kEpiThreads);
    }
    mbar_init(smem_u32(&B.drain), 1);
    B.abort = 0;
    fence_mbar_init();
  }
  // resident operands: W1 and W2 (already in operand order) and the biases
  {
    const uint4 *w1 = reinterpret_cast<const uint4 *>(W1p), *w2 = reinterpret_cast<const uint4 *>(W2p);
    uint4 *d1 = reinterpret_cast<uint4 *>(smem + L.w1), *d2 = reinterpret_cast<uint4 *>(smem + L.w2);
    const int n1 = H * D / 8, n2v = n2 * H / 8;
    for (int i = tid; i < n1; i += kTcThreads) d1[i] = __ldg(w1 + i);
    for (int i = tid; i < n2v; i += kTcThreads) d2[i] = __ldg(w2 + i);
  }
  for (int i = tid; i < H; i += kTcThreads) sb1[i] = b1[i];
  if (tid < 32) sb2[tid] = tid < b ? b2[tid] : 0.0f;
  fence_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = B.tmem_slot;

  if (warp == kWarpMma) {
    if (lane == 0) {
      const uint32_t idesc1 = mma_idesc(kRows, kHC), idesc2 = mma_idesc(kRows, n2);
      const uint32_t sx = sbase + L.x, sw1 = sbase + L.w1, sw2 = sbase + L.w2;
      // layer 2 of chunk number gp (chunk cp of tile number ip of this CTA):
      // hidden chunk (TMEM) x W2 chunk into the tile's accumulator
      auto layer2 = [&](uint32_t gp, uint32_t ip, int cp) -> bool {
        const int hb = (int)(gp & 1);
        if (!wait_or_abort(smem_u32(&B.hfull[hb]), (gp >> 1) & 1u, abort, wait_ns)) return false;
        if (cp == 0 && !wait_or_abort(smem_u32(&B.a2empty[ip & 1]), ((ip >> 1) & 1u) ^ 1u, abort, wait_ns))
          return false;
        tc_fence_after();
        const uint32_t d2 = tmem + kTmemAcc2 + (ip & 1u) * 32u;
        const uint32_t ah = tmem + kTmemHid + (uint32_t)hb * (kHC / 2);
        for (int ks = 0; ks < kHC / 16; ++ks)
          tc_mma_f16_ts(d2, ah + (uint32_t)ks * 8u,
                        smem_desc(sw2 + (uint32_t)cp * w2_bytes + ks * 256, 128, 16 * 128), idesc2,
                        (cp > 0 || ks > 0) ? 1u : 0u);
        tc_commit(smem_u32(&B.hempty[hb]));
        if (cp == nc - 1) tc_commit(smem_u32(&B.a2full[ip & 1]));
        return true;
      };
      bool ok = true;
      uint32_t g = 0, it = 0;  // chunks and tiles of this CTA so far
      for (int64_t tile = blockIdx.x; tile < ntiles && ok; tile += gridDim.x, ++it) {
        const int xb = nxb == 2 ? (int)(it & 1) : 0;
        const uint32_t xpar = (nxb == 2 ? it >> 1 : it) & 1u;
        if (!wait_or_abort(smem_u32(&B.xfull[xb]), xpar, abort, wait_ns)) {
          ok = false;
          break;
        }
        for (int c = 0; c < nc; ++c, ++g) {
          const int a = (int)(g & 1);
          if (!wait_or_abort(smem_u32(&B.a1empty[a]), ((g >> 1) & 1u) ^ 1u, abort, wait_ns)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d1 = tmem + (uint32_t)a * kHC;
          for (int ks = 0; ks < D / 16; ++ks)
            tc_mma_f16(d1, smem_desc(sx + (uint32_t)xb * x_bytes + ks * 256, 128, kx * 128),
                       smem_desc(sw1 + (uint32_t)c * w1_bytes + ks * 256, 128, kx * 128), idesc1,
                       ks > 0 ? 1u : 0u);
          tc_commit(smem_u32(&B.a1full[a]));
          if (c == nc - 1) tc_commit(smem_u32(&B.xempty[xb]));
          if (g > 0 && !layer2(g - 1, c > 0 ? it : it - 1, c > 0 ? c - 1 : nc - 1)) {
            ok = false;
            break;
          }
        }
      }
      if (ok && g > 0) layer2(g - 1, it - 1, nc - 1);
      // every MMA of this thread completes before TMEM is freed
      tc_commit(smem_u32(&B.drain));
      mbar_wait_bounded(smem_u32(&B.drain), 0);
    }
    __syncwarp();
  } else if (warp < kWarpConv) {
    const int lg = warp & 3;                 // TMEM lane group this warp may access
    const int hh = (warp - kWarpEpi) >> 2;   // column half of each chunk
    const int r = lg * 32 + lane;            // tile row = TMEM lane
    const uint32_t lane_base = (uint32_t)(lg * 32) << 16;
    const __half2 zero2 = __float2half2_rn(0.0f);
    // logits of tile number ip (global tile t): layer-2 accumulator + b2 -> out,
    // 16 columns a thread (its row, its column half), as float4 where aligned
    auto logits = [&](uint32_t ip, int64_t t) -> bool {
      if (!warp_wait(smem_u32(&B.a2full[ip & 1]), (ip >> 1) & 1u, abort, wait_ns)) return false;
      tc_fence_after();
      uint32_t o[16];
      const bool reads = hh * 16 < n2;  // same for the whole warp
      if (reads) {
        tc_ld16(tmem + lane_base + kTmemAcc2 + (ip & 1u) * 32u + (uint32_t)hh * 16u, o);
        tc_wait_ld();
      }
      tc_fence_before();
      mbar_arrive(smem_u32(&B.a2empty[ip & 1]));
      const int64_t row = t * kRows + r;
      const int ncol = b - hh * 16 < 16 ? b - hh * 16 : 16;
      if (reads && row < nq) {
        float *dst = out + row * b + hh * 16;
        const float *bias = sb2 + hh * 16;
        if (vec_out) {
#pragma unroll
          for (int q = 0; q < 4; ++q)
            if (4 * q < ncol)
              *reinterpret_cast<float4 *>(dst + 4 * q) =
                  make_float4(__fadd_rn(__uint_as_float(o[4 * q]), bias[4 * q]),
                              __fadd_rn(__uint_as_float(o[4 * q + 1]), bias[4 * q + 1]),
                              __fadd_rn(__uint_as_float(o[4 * q + 2]), bias[4 * q + 2]),
                              __fadd_rn(__uint_as_float(o[4 * q + 3]), bias[4 * q + 3]));
        } else {
#pragma unroll
          for (int j = 0; j < 16; ++j)
            if (j < ncol) dst[j] = __fadd_rn(__uint_as_float(o[j]), bias[j]);
        }
      }
      return true;
    };
    uint32_t g = 0, it = 0;
    int64_t last_tile = 0;
    bool ok = true;
    for (int64_t tile = blockIdx.x; tile < ntiles && ok; tile += gridDim.x, ++it) {
      for (int c = 0; c < nc; ++c, ++g) {
        const int a = (int)(g & 1);
        if (!warp_wait(smem_u32(&B.a1full[a]), (g >> 1) & 1u, abort, wait_ns)) {
          ok = false;
          break;
        }
        tc_fence_after();
        // h = ReLU(s acc + b1) as fp16 pairs, 32 accumulator columns at a time
        const uint32_t col = tmem + lane_base + (uint32_t)a * kHC + (uint32_t)hh * 64u;
        const float *bb = sb1 + c * kHC + hh * 64;
        // both 32-column loads in flight before one wait
        uint32_t v[64];
        tc_ld32(col, *reinterpret_cast<uint32_t(*)[32]>(&v[0]));
        tc_ld32(col + 32u, *reinterpret_cast<uint32_t(*)[32]>(&v[32]));
        tc_wait_ld();
        uint32_t hp[32];
#pragma unroll
        for (int j4 = 0; j4 < 16; ++j4) {
          const float4 bq = reinterpret_cast<const float4 *>(bb)[j4];
          const float h0 = __fmaf_rn(s, __uint_as_float(v[4 * j4]), bq.x);
          const float h1 = __fmaf_rn(s, __uint_as_float(v[4 * j4 + 1]), bq.y);
          const float h2 = __fmaf_rn(s, __uint_as_float(v[4 * j4 + 2]), bq.z);
          const float h3 = __fmaf_rn(s, __uint_as_float(v[4 * j4 + 3]), bq.w);
          const __half2 p0 = __hmax2(__floats2half2_rn(h0, h1), zero2);
          const __half2 p1 = __hmax2(__floats2half2_rn(h2, h3), zero2);
          hp[2 * j4] = *reinterpret_cast<const uint32_t *>(&p0);
          hp[2 * j4 + 1] = *reinterpret_cast<const uint32_t *>(&p1);
        }
        tc_fence_before();
        mbar_arrive(smem_u32(&B.a1empty[a]));
        // the layer-2 MMAs of chunk g - 2 have read this hidden buffer
        if (!warp_wait(smem_u32(&B.hempty[a]), ((g >> 1) & 1u) ^ 1u, abort, wait_ns)) {
          ok = false;
          break;
        }
        tc_fence_after();
        tc_st32(tmem + lane_base + kTmemHid + (uint32_t)a * (kHC / 2) + (uint32_t)hh * 32u, hp);
        tc_wait_st();
        tc_fence_before();
        mbar_arrive(smem_u32(&B.hfull[a]));
        // the previous tile's logits, once this tile's first chunk is on its way
        if (c == 0 && it > 0 && !logits(it - 1, last_tile)) {
          ok = false;
          break;
        }
      }
      last_tile = tile;
      if (!ok) break;
    }
    if (ok && it > 0) ok = logits(it - 1, last_tile);
  } else {
    tc_convert_tiles<DT>(x, D, kx, nxb, nq, ntiles, x_bytes, smem + L.x, B.xfull, B.xempty, abort,
                         wait_ns, tid - kWarpConv * 32);
  }
  tc_fence_before();
  __syncthreads();
  if (tid == 0 && B.abort) atomicCAS(err, 0, NR_DEV_TIMEOUT);
  if (warp == kWarpMma) {
    tc_fence_after();
    tc_dealloc(tmem, kTmemCols);
  }
}

// ------------------------------------------------------------ one layer on tensor cores
// Encoders with hidden layers after the first run layer by layer, each layer
// y = act(s x W^T + b) as a persistent tensor-core GEMM: a CTA takes
// (128-row tile, Nt-column tile) items; producers fill a ring of kLyStages
// shared-memory stages with 64-wide K slices of x and of W; one thread issues
// four tcgen05.mma (K = 16 each) a slice into one of two TMEM accumulators;
// four epilogue warps (one per TMEM lane group) read it back, apply s, the
// bias and ReLU (hidden layers) and write fp16 activations, or fp32 logits
// for the last layer.
//
// W sits in global memory as (Npad / Nt) column tiles x (K / 64) slices of
// Nt x 64 fp16 in the K-major core-matrix order (the host writes it so at
// load), and hidden activations are written in the same order, as 128-row
// tiles x 64-column slices of 16 KB: every slice of either operand is one
// contiguous block, fetched by one bulk copy (cp.async.bulk, completing on
// an mbarrier by its byte count). The first layer's input is converted to
// fp16 by two groups of four producer warps, which take alternate slices:
// fp32 rows arrive by 2D tensor copies (cp.async.bulk.tensor, a warp of
// their own, 128-byte swizzle) in a ring of raw stages that the producers
// read from shared memory; uint8 rows go through the producers' registers.
// Each group's first thread fetches W for its slices. Waits are bounded as in
// the kernel above; a CTA that gives up first waits (bounded) for the bulk
// and tensor copies it issued.
constexpr int kLyKs = 64;        // K elements a slice
constexpr int kLyStages = 3;
// slices g and g + kLyPeriod use the same stage and the same producer group
constexpr int kLyPeriod = kLyStages % 2 == 0 ? kLyStages : 2 * kLyStages;
constexpr int kLyRawMax = 4;     // raw fp32 stages (first layer), at most
constexpr uint32_t kLyRawStage = (uint32_t)kRows * kLyKs * 4u;  // 32 KB: two 16 KB boxes
constexpr int kLyEpiWarps = 4, kLyProdWarps = 4;  // a producer group
constexpr int kLyWarpEpi = 1, kLyWarpProd = kLyWarpEpi + kLyEpiWarps;
constexpr int kLyWarpTma = kLyWarpProd + 2 * kLyProdWarps;
constexpr int kLyThreads = 32 * (kLyWarpTma + 1);  // 448
constexpr int kLyProdThreads = 32 * kLyProdWarps, kLyEpiThreads = 32 * kLyEpiWarps;
constexpr uint32_t kLyXSlice = (uint32_t)kRows * kLyKs * 2u;    // 16 KB of fp16

struct LyBars {
  uint64_t xfull[kLyStages];  // x stored by the producer threads (first layer)
  uint64_t tfull[2][kLyStages];  // a producer group's bulk copies into the stage landed
  uint64_t empty[kLyStages];
  uint64_t rawfull[kLyRawMax], rawempty[kLyRawMax];  // fp32 rows by tensor copy (first layer)
  uint64_t accfull[2], accempty[2];
  uint64_t drain;
  uint32_t tmem_slot;
  int abort;
};

__host__ __device__ inline uint32_t ly_stage_bytes(int Nt) { return kLyXSlice + (uint32_t)Nt * kLyKs * 2u; }
// operand stages, the bars, then (fp32 first layer) nraw raw stages from the
// next 1024-byte boundary (the 128-byte swizzle's alignment)
__host__ __device__ inline uint32_t ly_smem_bytes(int Nt, int nraw) {
  return kLyStages * ly_stage_bytes(Nt) + (uint32_t)sizeof(LyBars) +
         (nraw > 0 ? 1024u + (uint32_t)nraw * kLyRawStage : 0u);
}
// TMEM columns of the two accumulators: a power of two of at least 32
__host__ __device__ inline uint32_t ly_tmem_cols(int Nt) {
  uint32_t c = 32;
  while (c < 2u * (uint32_t)Nt) c <<= 1;
  return c;
}

__device__ __forceinline__ void mbar_arrive_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;\n" ::"r"(bar), "r"(bytes)
               : "memory");
}
// 2D tensor copy global -> this CTA's shared memory (box of the tensor map at
// element coordinates (c0, c1)), completing on `bar` by bytes
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *tm, int c0, int c1, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];\n" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tm)), "r"(c0), "r"(c1), "r"(bar)
      : "memory");
}
// bulk copy global -> this CTA's shared memory, completing on `bar` by bytes
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void *src, uint32_t bytes, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];\n" ::"r"(dst),
      "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}

// XT: the input's type (0 uint8 rows, 1 fp32 rows, 2 fp16 activations in
// operand order); YF: 1 fp32 output rows (the logits, no activation), 0 fp16
// activations in operand order with ReLU. x [n x K], y [n x N].
template <int XT, int YF>
__global__ void __launch_bounds__(kLyThreads, 1)
    encode_layer_kernel(const void *__restrict__ x, int K, int N, int Nt, int Npad, float s,
                        const __half *__restrict__ Wp, const float *__restrict__ bias, int64_t n,
                        void *__restrict__ y, int nraw, const __grid_constant__ CUtensorMap tmx,
                        int *err, int64_t wait_ns) {
  extern __shared__ __align__(1024) unsigned char smem[];
  const uint32_t stage_b = ly_stage_bytes(Nt);
  LyBars &B = *reinterpret_cast<LyBars *>(smem + kLyStages * stage_b);
  // raw stages (XT 1): nraw x 32 KB from the first 1024-byte boundary after the bars
  const uint32_t raw_s =
      (smem_u32(smem) + kLyStages * stage_b + (uint32_t)sizeof(LyBars) + 1023u) & ~1023u;
  const unsigned char *raw = smem + (raw_s - smem_u32(smem));
  volatile int *abort = &B.abort;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nks = K / kLyKs;                       // slices an item
  const int nct = Npad / Nt;                       // column tiles
  const int64_t nrt = (n + kRows - 1) / kRows;     // row tiles
  const int64_t items = nrt * nct;
  const uint32_t sbase = smem_u32(smem);
  const uint32_t tcols = ly_tmem_cols(Nt);
  const uint32_t wbytes = (uint32_t)Nt * kLyKs * 2u;
  if (warp == 0) {
    tc_alloc(smem_u32(&B.tmem_slot), tcols);
    tc_relinquish();
  }
  if (tid == 0) {
    for (int i = 0; i < kLyStages; ++i) {
      mbar_init(smem_u32(&B.xfull[i]), kLyProdThreads);
      mbar_init(smem_u32(&B.tfull[0][i]), 1);
      mbar_init(smem_u32(&B.tfull[1][i]), 1);
      mbar_init(smem_u32(&B.empty[i]), 1);
    }
    for (int i = 0; i < kLyRawMax; ++i) {
      mbar_init(smem_u32(&B.rawfull[i]), 1);
      mbar_init(smem_u32(&B.rawempty[i]), kLyProdThreads);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&B.accfull[i]), 1);
      mbar_init(smem_u32(&B.accempty[i]), kLyEpiThreads);
    }
    mbar_init(smem_u32(&B.drain), 1);
    B.abort = 0;
    fence_mbar_init();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = B.tmem_slot;

  if (warp == kLyWarpTma) {
    // fp32 first layer: lane 0 fetches each slice's 128 rows x 64 values by
    // two tensor copies (boxes of 32 values x 128 rows, 128-byte swizzle;
    // rows past n read as zeros) into raw stage g % nraw
    if (XT == 1 && lane == 0) {
      uint32_t g = 0;
      bool ok = true;
      for (int64_t item = blockIdx.x; item < items && ok; item += gridDim.x) {
        const int row0 = (int)(item / nct * kRows);
        for (int ks = 0; ks < nks; ++ks, ++g) {
          const uint32_t rs = g % (uint32_t)nraw;
          if (!wait_or_abort(smem_u32(&B.rawempty[rs]), ((g / (uint32_t)nraw) & 1u) ^ 1u, abort, wait_ns)) {
            ok = false;
            break;
          }
          const uint32_t bar = smem_u32(&B.rawfull[rs]), dst = raw_s + rs * kLyRawStage;
          mbar_arrive_tx(bar, kLyRawStage);
          tma_load_2d(dst, &tmx, ks * kLyKs, row0, bar);
          tma_load_2d(dst + kLyRawStage / 2, &tmx, ks * kLyKs + kLyKs / 2, row0, bar);
        }
      }
      // the copies issued (the last on each stage are among the last nraw) land
      // before the CTA ends, even if a role gave up
      for (uint32_t i = g > (uint32_t)nraw ? g - nraw : 0u; i < g; ++i)
        mbar_wait_bounded(smem_u32(&B.rawfull[i % nraw]), (i / nraw) & 1u);
    }
    __syncwarp();
  } else if (warp == 0) {
    if (lane == 0) {  // the MMA thread
      const uint32_t idesc = mma_idesc(kRows, Nt);
      uint32_t g = 0, it = 0;  // slices and items of this CTA so far
      bool ok = true;
      for (int64_t item = blockIdx.x; item < items && ok; item += gridDim.x, ++it) {
        const uint32_t a = it & 1u;
        if (!wait_or_abort(smem_u32(&B.accempty[a]), ((it >> 1) & 1u) ^ 1u, abort, wait_ns)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + a * (uint32_t)Nt;
        for (int ks = 0; ks < nks; ++ks, ++g) {
          const uint32_t st = g % kLyStages, ph = (g / kLyStages) & 1u;
          // the copies of slice g: group g % 2 (XT 0 / 1: that group's phases
          // on the stage are slices g, g + kLyPeriod, ...), or group 0 (XT 2)
          const uint32_t tb = XT == 2 ? smem_u32(&B.tfull[0][st]) : smem_u32(&B.tfull[g & 1u][st]);
          const uint32_t tph = XT == 2 ? ph : (g / kLyPeriod) & 1u;
          if (!wait_or_abort(tb, tph, abort, wait_ns) ||
              (XT != 2 && !wait_or_abort(smem_u32(&B.xfull[st]), ph, abort, wait_ns))) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sx = sbase + st * stage_b, sw = sx + kLyXSlice;
          for (int k = 0; k < kLyKs / 16; ++k)
            tc_mma_f16(d, smem_desc(sx + (uint32_t)k * 256u, 128, 8 * 128),
                       smem_desc(sw + (uint32_t)k * 256u, 128, 8 * 128), idesc,
                       (ks > 0 || k > 0) ? 1u : 0u);
          tc_commit(smem_u32(&B.empty[st]));
        }
        if (!ok) break;
        tc_commit(smem_u32(&B.accfull[a]));
      }
      // every MMA of this thread completes before TMEM is freed
      tc_commit(smem_u32(&B.drain));
      mbar_wait_bounded(smem_u32(&B.drain), 0);
    }
    __syncwarp();
  } else if (warp < kLyWarpProd) {  // epilogue: one TMEM lane group a warp
    const int lg = warp & 3;
    const uint32_t lane_base = (uint32_t)(lg * 32) << 16;
    const int r = lg * 32 + lane;  // the row in the tile
    uint32_t it = 0;
    for (int64_t item = blockIdx.x; item < items; item += gridDim.x, ++it) {
      const uint32_t a = it & 1u;
      if (!warp_wait(smem_u32(&B.accfull[a]), (it >> 1) & 1u, abort, wait_ns)) break;
      tc_fence_after();
      const int64_t rt = item / nct;
      const int c0 = (int)(item % nct) * Nt;
      const int64_t row = rt * kRows + r;
      for (int cc = 0; cc < Nt; cc += 32) {
        uint32_t v[32];
        if (Nt - cc >= 32) {
          tc_ld32(tmem + lane_base + a * (uint32_t)Nt + (uint32_t)cc, v);
        } else {
          uint32_t w16[16];
          tc_ld16(tmem + lane_base + a * (uint32_t)Nt + (uint32_t)cc, w16);
#pragma unroll
          for (int j = 0; j < 16; ++j) v[j] = w16[j];
        }
        tc_wait_ld();
        const int ncol = min(32, Nt - cc);
        if (row < n) {
          if (YF) {
            float *dst = static_cast<float *>(y) + row * N;
#pragma unroll
            for (int j = 0; j < 32; ++j) {
              const int col = c0 + cc + j;
              if (j < ncol && col < N) dst[col] = __fmaf_rn(s, __uint_as_float(v[j]), bias[col]);
            }
          } else {
            // hidden widths are multiples of 64: every column of the tile
            // exists; 8 columns (16 bytes) go to their core-matrix row
            __half *tile = static_cast<__half *>(y) + (size_t)rt * N * kRows;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              if (8 * q >= ncol) break;
              const int col = c0 + cc + 8 * q;
              uint32_t hp[4];
#pragma unroll
              for (int j = 0; j < 4; ++j) {
                const float h0 = __fmaf_rn(s, __uint_as_float(v[8 * q + 2 * j]), bias[col + 2 * j]);
                const float h1 = __fmaf_rn(s, __uint_as_float(v[8 * q + 2 * j + 1]), bias[col + 2 * j + 1]);
                const __half2 p = __hmax2(__floats2half2_rn(h0, h1), __float2half2_rn(0.0f));
                hp[j] = *reinterpret_cast<const uint32_t *>(&p);
              }
              __half *dst = tile + (size_t)(col >> 6) * (kRows * kLyKs) +
                            nr_tc_kmajor_off(r, (col & 63) >> 3, 8) / 2;
              *reinterpret_cast<uint4 *>(dst) = make_uint4(hp[0], hp[1], hp[2], hp[3]);
            }
          }
        }
      }
      tc_fence_before();
      mbar_arrive(smem_u32(&B.accempty[a]));
    }
  } else if (warp < kLyWarpTma) {  // producers: x and W slices into the stage ring
    const int grp = (warp - kLyWarpProd) / kLyProdWarps;  // XT 0 / 1: two groups
    const int ct = tid - kLyWarpProd * 32 - grp * kLyProdThreads;
    const bool lead = ct == 0;  // issues the bulk copies (of its group's slices)
    uint32_t g = 0;
    bool ok = true;
    for (int64_t item = blockIdx.x; item < items && ok; item += gridDim.x) {
      const int64_t rt = item / nct;
      const int ctile = (int)(item % nct);
      const int64_t row0 = rt * kRows;
      const int rows = n - row0 < kRows ? (int)(n - row0) : kRows;
      const char *wt = reinterpret_cast<const char *>(Wp) + (size_t)ctile * nks * wbytes;
      for (int ks = 0; ks < nks; ++ks, ++g) {
        const uint32_t st = g % kLyStages, ph = ((g / kLyStages) & 1u) ^ 1u;
        unsigned char *sx = smem + st * stage_b;
        if (XT == 2) {  // both operands by bulk copy, from one thread
          if (!lead || grp != 0) continue;
          if (!wait_or_abort(smem_u32(&B.empty[st]), ph, abort, wait_ns)) {
            ok = false;
            break;
          }
          const uint32_t bar = smem_u32(&B.tfull[0][st]);
          mbar_arrive_tx(bar, kLyXSlice + wbytes);
          bulk_g2s(sbase + st * stage_b,
                   static_cast<const char *>(x) + ((size_t)rt * nks + ks) * kLyXSlice, kLyXSlice, bar);
          bulk_g2s(sbase + st * stage_b + kLyXSlice, wt + (size_t)ks * wbytes, wbytes, bar);
          continue;
        }
        // group grp takes the slices g with g % 2 == grp: two slices' loads
        // in flight. Warp pw of the group takes rows 32 pw .. 32 pw + 31; in
        // each load a lane reads row 8 i + lane % 8 of them, so that a warp
        // touches 8 rows (8 cache lines) and every 8 lanes store 8 different
        // rows of one chunk (different banks in the core-matrix layout)
        if ((g & 1u) != (uint32_t)grp) continue;
        const int pw = ct >> 5, rl = lane & 7, q = lane >> 3;
        uint4 xv[8];
        if (XT == 1) {
          // from raw stage g % nraw: value column 8 c + 4 h of row r sits in
          // box c / 4, 16-byte piece (2 (c % 4) + h) ^ (r % 8) of the row's
          // 128 bytes (the swizzle; 8 lanes read 8 rows, different banks)
          const uint32_t rs = g % (uint32_t)nraw;
          if (!warp_wait(smem_u32(&B.rawfull[rs]), (g / (uint32_t)nraw) & 1u, abort, wait_ns)) {
            ok = false;
            break;
          }
          const unsigned char *rst = raw + rs * kLyRawStage;
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const int r = pw * 32 + 8 * i + rl;
#pragma unroll
            for (int jj = 0; jj < 2; ++jj) {  // chunk q + 4 jj: box jj, pieces 2q, 2q + 1
              const unsigned char *row = rst + jj * (kLyRawStage / 2) + r * 128;
              const float4 u = *reinterpret_cast<const float4 *>(row + (((2 * q) ^ (r & 7)) << 4));
              const float4 w = *reinterpret_cast<const float4 *>(row + (((2 * q + 1) ^ (r & 7)) << 4));
              const __half2 h0 = __floats2half2_rn(u.x, u.y), h1 = __floats2half2_rn(u.z, u.w);
              const __half2 h2 = __floats2half2_rn(w.x, w.y), h3 = __floats2half2_rn(w.z, w.w);
              xv[2 * i + jj] = make_uint4(*reinterpret_cast<const uint32_t *>(&h0),
                                          *reinterpret_cast<const uint32_t *>(&h1),
                                          *reinterpret_cast<const uint32_t *>(&h2),
                                          *reinterpret_cast<const uint32_t *>(&h3));
            }
          }
          mbar_arrive(smem_u32(&B.rawempty[rs]));
        } else {
#pragma unroll
          for (int i = 0; i < 4; ++i) {  // 16 uint8 values (piece q) -> chunks 2q, 2q + 1
            const int r = pw * 32 + 8 * i + rl;
            uint4 v = make_uint4(0u, 0u, 0u, 0u);
            if (r < rows)
              v = __ldg(reinterpret_cast<const uint4 *>(static_cast<const uint8_t *>(x) + (row0 + r) * K +
                                                        ks * kLyKs) + q);
            u8x16_to_f16(v, xv[2 * i], xv[2 * i + 1]);
          }
        }
        if (!warp_wait(smem_u32(&B.empty[st]), ph, abort, wait_ns)) {
          ok = false;
          break;
        }
        if (lead) {
          const uint32_t bar = smem_u32(&B.tfull[grp][st]);
          mbar_arrive_tx(bar, wbytes);
          bulk_g2s(sbase + st * stage_b + kLyXSlice, wt + (size_t)ks * wbytes, wbytes, bar);
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int r = pw * 32 + 8 * i + rl;
#pragma unroll
          for (int jj = 0; jj < 2; ++jj) {
            const int c = XT == 1 ? q + 4 * jj : 2 * q + jj;
            *reinterpret_cast<uint4 *>(sx + nr_tc_kmajor_off(r, c, 8)) = xv[2 * i + jj];
          }
        }
        fence_async_smem();
        mbar_arrive(smem_u32(&B.xfull[st]));
      }
    }
    // the bulk copies it issued land before the CTA ends, even if a role
    // gave up: the latest phase of each of its barriers (XT 2: slices
    // g - kLyStages .. g - 1, all group 0's; else its slices among
    // g - kLyPeriod .. g - 1)
    if (lead) {
      if (XT == 2) {
        if (grp == 0)
          for (uint32_t i = g > (uint32_t)kLyStages ? g - kLyStages : 0u; i < g; ++i)
            mbar_wait_bounded(smem_u32(&B.tfull[0][i % kLyStages]), (i / kLyStages) & 1u);
      } else {
        for (uint32_t i = g > (uint32_t)kLyPeriod ? g - kLyPeriod : 0u; i < g; ++i)
          if ((i & 1u) == (uint32_t)grp)
            mbar_wait_bounded(smem_u32(&B.tfull[grp][i % kLyStages]), (i / kLyPeriod) & 1u);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (tid == 0 && B.abort) atomicCAS(err, 0, NR_DEV_TIMEOUT);
  if (warp == 0) {
    tc_fence_after();
    tc_dealloc(tmem, tcols);
  }
}

// X tile buffers for a shape: 2 if a block's shared memory allows, else 1, else 0
int tc_xbuffers(int D, int H, int n2, int smem_optin) {
  for (int nxb = 2; nxb >= 1; --nxb)
    if (tc_layout(D, H, n2, nxb).total <= (uint32_t)smem_optin) return nxb;
  return 0;
}

// ------------------------------------------------------------ CUDA-core kernel
constexpr int kQB = 8;
constexpr int kThreads = 256;

__global__ void __launch_bounds__(kThreads)
    encode_simt_kernel(const void *__restrict__ x, int dtype, int D, int H, int b, float s,
                       const float *__restrict__ W1T, const float *__restrict__ b1,
                       const float *__restrict__ W2, const float *__restrict__ b2, int64_t nq,
                       float *__restrict__ out) {
  extern __shared__ float sm[];
  float *xs = sm;                    // [kQB][D]
  float *hs = sm + (size_t)kQB * D;  // [kQB][H]
  const int tid = threadIdx.x;
  const int64_t q0 = (int64_t)blockIdx.x * kQB;
  for (int i = tid; i < kQB * D; i += kThreads) {
    const int qi = i / D, j = i - qi * D;
    const int64_t qq = q0 + qi;
    float v = 0.0f;
    if (qq < nq)
      v = dtype == 0 ? (float)static_cast<const uint8_t *>(x)[qq * D + j]
                     : static_cast<const float *>(x)[qq * D + j];
    xs[i] = v;
  }
  __syncthreads();
  for (int u = tid; u < H; u += kThreads) {
    float acc[kQB];
#pragma unroll
    for (int qi = 0; qi < kQB; ++qi) acc[qi] = 0.0f;
    for (int j = 0; j < D; ++j) {
      const float w = W1T[(size_t)j * H + u];
#pragma unroll
      for (int qi = 0; qi < kQB; ++qi) acc[qi] = __fmaf_rn(w, xs[qi * D + j], acc[qi]);
    }
#pragma unroll
    for (int qi = 0; qi < kQB; ++qi) {
      const float h = __fmaf_rn(s, acc[qi], b1[u]);
      hs[qi * H + u] = h > 0.0f ? h : 0.0f;
    }
  }
  __syncthreads();
  for (int o = tid; o < kQB * b; o += kThreads) {
    const int qi = o / b, j = o - qi * b;
    const int64_t qq = q0 + qi;
    if (qq >= nq) continue;
    float acc = b2[j];
    const float *w = W2 + (size_t)j * H;
    for (int u = 0; u < H; ++u) acc = __fmaf_rn(w[u], hs[qi * H + u], acc);
    out[qq * b + j] = acc;
  }
}

// Encoders with hidden layers after the first: kQB queries a block, every
// layer's activations for them in shared memory (two buffers of kQB x the
// widest layer), one thread per output unit; layer weights transposed
// [previous x width] so that a warp's loads are contiguous.
__global__ void __launch_bounds__(kThreads)
    encode_mlp_kernel(const void *__restrict__ x, int dtype, int D, int H, int b, float s,
                      const float *__restrict__ W1T, const float *__restrict__ b1, int n_mid,
                      int4 mid_lo, int4 mid_hi, const float *__restrict__ WmT,
                      const float *__restrict__ W2, const float *__restrict__ b2, int maxw,
                      int64_t nq, float *__restrict__ out) {
  extern __shared__ float sm[];
  float *A = sm, *B = sm + (size_t)kQB * maxw;  // [kQB][width] each
  const int tid = threadIdx.x;
  const int64_t q0 = (int64_t)blockIdx.x * kQB;
  for (int i = tid; i < kQB * D; i += kThreads) {
    const int qi = i / D, j = i - qi * D;
    const int64_t qq = q0 + qi;
    float v = 0.0f;
    if (qq < nq)
      v = dtype == 0 ? (float)static_cast<const uint8_t *>(x)[qq * D + j]
                     : static_cast<const float *>(x)[qq * D + j];
    A[qi * D + j] = v;
  }
  __syncthreads();
  for (int u = tid; u < H; u += kThreads) {  // first hidden layer, input scale s
    float acc[kQB];
#pragma unroll
    for (int qi = 0; qi < kQB; ++qi) acc[qi] = 0.0f;
    for (int j = 0; j < D; ++j) {
      const float w = W1T[(size_t)j * H + u];
#pragma unroll
      for (int qi = 0; qi < kQB; ++qi) acc[qi] = __fmaf_rn(w, A[qi * D + j], acc[qi]);
    }
#pragma unroll
    for (int qi = 0; qi < kQB; ++qi) {
      const float h = __fmaf_rn(s, acc[qi], b1[u]);
      B[qi * H + u] = h > 0.0f ? h : 0.0f;
    }
  }
  __syncthreads();
  const int widths[8] = {mid_lo.x, mid_lo.y, mid_lo.z, mid_lo.w, mid_hi.x, mid_hi.y, mid_hi.z, 0};
  int prev = H;
  const float *wl = WmT;
  float *cur = B, *nxt = A;
  for (int l = 0; l < n_mid; ++l) {
    const int w = widths[l];
    const float *bias = wl + (size_t)w * prev;
    for (int u = tid; u < w; u += kThreads) {
      float acc[kQB];
#pragma unroll
      for (int qi = 0; qi < kQB; ++qi) acc[qi] = bias[u];
      for (int j = 0; j < prev; ++j) {
        const float wj = wl[(size_t)j * w + u];
#pragma unroll
        for (int qi = 0; qi < kQB; ++qi) acc[qi] = __fmaf_rn(wj, cur[qi * prev + j], acc[qi]);
      }
#pragma unroll
      for (int qi = 0; qi < kQB; ++qi) nxt[qi * w + u] = acc[qi] > 0.0f ? acc[qi] : 0.0f;
    }
    __syncthreads();
    wl = bias + w;
    prev = w;
    float *t = cur;
    cur = nxt;
    nxt = t;
  }
  for (int o = tid; o < kQB * b; o += kThreads) {  // last layer, linear
    const int qi = o / b, j = o - qi * b;
    const int64_t qq = q0 + qi;
    if (qq >= nq) continue;
    float acc = b2[j];
    const float *w = W2 + (size_t)j * prev;
    for (int u = 0; u < prev; ++u) acc = __fmaf_rn(w[u], cur[qi * prev + u], acc);
    out[qq * b + j] = acc;
  }
}

}  // namespace

bool nr_encode_uses_tensor_cores(const nr_index *ix) {
  if (ix->n_ly > 0) return true;
  return ix->W1h != nullptr && ix->n_mid == 0 && ix->D % 16 == 0 && ix->D <= 128 &&
         ix->H % kHC == 0 && ix->b <= 32 &&
         tc_xbuffers(ix->D, ix->H, ix->b <= 16 ? 16 : 32, ix->smem_optin) > 0;
}

// rows a layer-by-layer encode runs at once (its activation scratch: two
// buffers of rows x the widest hidden layer, fp16)
constexpr int64_t kEncRowBlock = (int64_t)1 << 18;

static int enc_max_hidden(const nr_index *ix) {
  int m = ix->H;
  for (int l = 0; l < ix->n_mid; ++l) m = ix->mid_w[l] > m ? ix->mid_w[l] : m;
  return m;
}

size_t nr_encode_scratch_bytes(const nr_index *ix, int64_t n) {
  if (ix->n_ly == 0 || n <= 0) return 0;
  // whole 128-row tiles: the bulk copies of a ragged last tile stay in the buffer
  const int64_t rows = ((n < kEncRowBlock ? n : kEncRowBlock) + kRows - 1) / kRows * kRows;
  return ((size_t)rows * enc_max_hidden(ix) * 2 + 255) / 256 * 256 * 2;
}

// The driver's tensor-map encoder, looked up once through the runtime (so the
// library needs no link-time dependency on the driver library).
static PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess) {
      cudaGetLastError();
      p = nullptr;
    }
    return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }();
  return fn;
}

template <int XT, int YF>
static cudaError_t launch_layer(nr_index *ix, const void *x, int K, int N, int l, float sc,
                                const float *bias, int64_t n, void *y, int64_t wait_ns,
                                cudaStream_t s) {
  const int nt = ix->ly_nt[l], Np = (N + 15) / 16 * 16;
  // fp32 first layer: raw stages for the tensor copies, as many as fit (<= 4)
  int nraw = 0;
  CUtensorMap tm;
  memset(&tm, 0, sizeof(tm));
  if (XT == 1) {
    nraw = kLyRawMax;
    while (nraw > 1 && ly_smem_bytes(nt, nraw) > (uint32_t)ix->smem_optin) --nraw;
    if (ly_smem_bytes(nt, nraw) > (uint32_t)ix->smem_optin) return cudaErrorInvalidConfiguration;
    // x [n rows x K] fp32: boxes of 32 values x 128 rows, 128-byte swizzle
    const cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)n};
    const cuuint64_t strides[1] = {(cuuint64_t)K * 4u};
    const cuuint32_t box[2] = {(cuuint32_t)(kLyKs / 2), (cuuint32_t)kRows}, es[2] = {1u, 1u};
    const PFN_cuTensorMapEncodeTiled_v12000 encode = tensor_map_encoder();
    if (!encode) return cudaErrorNotSupported;
    if (encode(&tm, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<void *>(x), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  uint32_t smem = ly_smem_bytes(nt, nraw);
  // accumulators wider than half of TMEM: one CTA an SM (a second would
  // stall in its TMEM allocation until the first ends)
  if (ly_tmem_cols(nt) > 256 && smem <= (uint32_t)ix->smem_optin / 2)
    smem = (uint32_t)ix->smem_optin / 2 + 1024;
  auto kern = encode_layer_kernel<XT, YF>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const int64_t items = (n + kRows - 1) / kRows * (Np / nt);
  const int64_t grid = items < ix->num_sms ? items : ix->num_sms;
  kern<<<(unsigned)grid, kLyThreads, smem, s>>>(x, K, N, nt, Np, sc,
                                                static_cast<const __half *>(ix->Wl) + ix->ly_off[l],
                                                bias, n, y, nraw, tm, ix->d_err, wait_ns);
  ix->launches += 1;
  return cudaGetLastError();
}

// An encoder with hidden layers after the first, layer by layer on tensor
// cores, in row blocks of kEncRowBlock (activations in scratch).
static cudaError_t encode_layers(nr_index *ix, const void *d_x, int64_t nq, float *d_logits,
                                 cudaStream_t s, void *scratch, int64_t wait_ns) {
  const int L = ix->n_ly;
  const size_t half = nr_encode_scratch_bytes(ix, nq) / 2;
  __half *act[2] = {static_cast<__half *>(scratch),
                    reinterpret_cast<__half *>(static_cast<char *>(scratch) + half)};
  const size_t esz = ix->dtype == 0 ? 1 : 4;
  for (int64_t r0 = 0; r0 < nq; r0 += kEncRowBlock) {
    const int64_t n = nq - r0 < kEncRowBlock ? nq - r0 : kEncRowBlock;
    const void *x = static_cast<const char *>(d_x) + (size_t)r0 * ix->D * esz;
    cudaError_t e = ix->dtype == 0
                        ? launch_layer<0, 0>(ix, x, ix->D, ix->H, 0, ix->in_scale, ix->b1, n, act[0],
                                             wait_ns, s)
                        : launch_layer<1, 0>(ix, x, ix->D, ix->H, 0, ix->in_scale, ix->b1, n, act[0],
                                             wait_ns, s);
    if (e != cudaSuccess) return e;
    size_t o = 0;  // the middle layers' weights then bias, as the file stores them
    int prev = ix->H;
    for (int l = 0; l < ix->n_mid; ++l) {
      const int w = ix->mid_w[l];
      const float *bias = ix->Wm + o + (size_t)w * prev;
      e = launch_layer<2, 0>(ix, act[l & 1], prev, w, l + 1, 1.0f, bias, n, act[(l + 1) & 1], wait_ns,
                             s);
      if (e != cudaSuccess) return e;
      o += (size_t)w * prev + w;
      prev = w;
    }
    e = launch_layer<2, 1>(ix, act[ix->n_mid & 1], prev, ix->b, L - 1, 1.0f, ix->b2, n,
                           d_logits + (size_t)r0 * ix->b, wait_ns, s);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

cudaError_t nr_launch_encode(nr_index *ix, const void *d_x, int64_t nq, float *d_logits,
                             cudaStream_t s, void *scratch) {
  if (nq <= 0) return cudaSuccess;
  const int wl = ix->params.wait_limit_us;
  const int64_t wait_ns = wl == 0 ? (int64_t)1000000000 : wl > 0 ? (int64_t)wl * 1000 : (int64_t)-1;
  if (ix->n_ly > 0 && (reinterpret_cast<uintptr_t>(d_x) & 15) == 0) {
    if (!scratch) {  // the index's own scratch, grown on demand
      const size_t need = nr_encode_scratch_bytes(ix, nq);
      if (ix->enc_ws_cap < need) {
        cudaError_t e = cudaDeviceSynchronize();  // earlier encodes may still read it
        if (e != cudaSuccess) return e;
        if (ix->enc_ws) cudaFree(ix->enc_ws);
        ix->enc_ws = nullptr;
        ix->enc_ws_cap = 0;
        e = cudaMalloc(&ix->enc_ws, need);
        if (e != cudaSuccess) return e;
        ix->enc_ws_cap = need;
      }
      scratch = ix->enc_ws;
    }
    return encode_layers(ix, d_x, nq, d_logits, s, scratch, wait_ns);
  }
  // the tensor-core kernel reads X in 16-byte pieces
  if (nr_encode_uses_tensor_cores(ix) && (reinterpret_cast<uintptr_t>(d_x) & 15) == 0) {
    const int n2 = ix->b <= 16 ? 16 : 32;
    const int nxb = tc_xbuffers(ix->D, ix->H, n2, ix->smem_optin);
    const uint32_t smem = tc_layout(ix->D, ix->H, n2, nxb).total;
    const int64_t tiles = (nq + kRows - 1) / kRows;
    const int64_t grid = tiles < ix->num_sms ? tiles : ix->num_sms;
    auto kern = ix->dtype == 0 ? encode_tc_kernel<0> : encode_tc_kernel<1>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int vec_out = ix->b % 4 == 0 && (reinterpret_cast<uintptr_t>(d_logits) & 15) == 0;
    // the roles' hand-off waits: wait_ns (1 s by default); the drain of
    // issued MMAs before TMEM is freed keeps its own 1 s bound whatever this is
    kern<<<(unsigned)grid, kTcThreads, smem, s>>>(d_x, ix->D, ix->H, ix->b, n2, nxb, vec_out, ix->in_scale,
                                                  static_cast<const __half *>(ix->W1h), ix->b1,
                                                  static_cast<const __half *>(ix->W2h), ix->b2, nq,
                                                  d_logits, ix->d_err, wait_ns);
    ix->launches += 1;
    return cudaGetLastError();
  }
  if (ix->n_mid > 0) {
    int maxw = ix->D > ix->H ? ix->D : ix->H;
    for (int i = 0; i < ix->n_mid; ++i) maxw = ix->mid_w[i] > maxw ? ix->mid_w[i] : maxw;
    const size_t smem = (size_t)2 * kQB * maxw * sizeof(float);
    cudaError_t e = cudaFuncSetAttribute(encode_mlp_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int *mw = ix->mid_w;
    const int64_t grid = (nq + kQB - 1) / kQB;
    encode_mlp_kernel<<<(unsigned)grid, kThreads, smem, s>>>(
        d_x, ix->dtype, ix->D, ix->H, ix->b, ix->in_scale, ix->W1T, ix->b1, ix->n_mid,
        make_int4(mw[0], mw[1], mw[2], mw[3]), make_int4(mw[4], mw[5], mw[6], 0), ix->WmT, ix->W2,
        ix->b2, maxw, nq, d_logits);
    ix->launches += 1;
    return cudaGetLastError();
  }
  const size_t smem = (size_t)kQB * (ix->D + ix->H) * sizeof(float);
  cudaError_t e = cudaFuncSetAttribute(encode_simt_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  const int64_t grid = (nq + kQB - 1) / kQB;
  encode_simt_kernel<<<(unsigned)grid, kThreads, smem, s>>>(d_x, ix->dtype, ix->D, ix->H, ix->b,
                                                             ix->in_scale, ix->W1T, ix->b1, ix->W2,
                                                             ix->b2, nq, d_logits);
  ix->launches += 1;
  return cudaGetLastError();
}
