// K1 encode: l = E(x), one hidden layer (Sec. 3.2.1):
//   h = ReLU(s (W1 x) + b1),  l = W2 h + b2.
//
// Tensor-core version (tcgen05, sm_103a). One CTA of 4 warps owns 128 query
// rows = the 128 TMEM lanes of its accumulators. Layer 1 runs in chunks of 128
// hidden units: one thread issues tcgen05.mma (kind::f16, fp16 operands, fp32
// accumulation in TMEM) over X [128 x D] and a W1 chunk [128 x D]; the four
// warps read the chunk back with tcgen05.ld, apply scale, bias and ReLU, and
// write it as fp16 into shared memory, where it becomes the A operand of the
// layer-2 MMA that accumulates l [128 x N2] (N2 = b padded to 16 or 32) in a
// second TMEM region across all chunks. Operands sit in shared memory in the
// canonical K-major no-swizzle layout (8-row x 16-byte core matrices; core
// matrices of one 8-row group consecutive along K). uint8 inputs are exact in
// fp16; the input scale is applied to the fp32 accumulator.
//
// Every wait on an MMA completion barrier is bounded (1 s); on timeout the
// kernel records NR_DEV_TIMEOUT, frees its TMEM and returns.
//
// Shapes the tensor-core kernel does not take (D % 16 != 0, D > 256,
// H % 128 != 0, b > 32) run on the CUDA-core kernel below it.
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

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

// byte offset of (row r, 16-byte K chunk c) in a K-major no-swizzle tile with
// kchunks chunks per row
__device__ __forceinline__ uint32_t kmajor_off(int r, int c, int kchunks) {
  return (uint32_t)((r & 7) * 16 + (r >> 3) * kchunks * 128 + c * 128);
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

constexpr int kRows = 128;  // query rows per CTA
constexpr int kHC = 128;    // hidden units per chunk
constexpr uint32_t kTmemCols = 256;

template <int DT>
__global__ void __launch_bounds__(128, 1)
    encode_tc_kernel(const void *__restrict__ x, int D, int H, int b, int n2, float s,
                     const __half *__restrict__ W1h, const float *__restrict__ b1,
                     const __half *__restrict__ W2h, const float *__restrict__ b2, int64_t nq,
                     float *__restrict__ out, int *err) {
  extern __shared__ __align__(1024) unsigned char smem[];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int kx = D / 8;  // 16-byte chunks per row of X and W1
  unsigned char *sX = smem;                            // [128][D] fp16
  unsigned char *sW1 = sX + kRows * D * 2;             // [128][D] fp16
  unsigned char *sH = sW1 + kHC * D * 2;               // [128][128] fp16
  unsigned char *sW2 = sH + kRows * kHC * 2;           // [n2][128] fp16
  float *sb1 = reinterpret_cast<float *>(sW2 + n2 * kHC * 2);  // [128]
  uint64_t *mbar = reinterpret_cast<uint64_t *>(sb1 + kHC);
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(mbar + 1);
  const uint32_t bar = smem_u32(mbar);
  const int64_t row0 = (int64_t)blockIdx.x * kRows;

  if (warp == 0) {
    tc_alloc(smem_u32(tmem_slot), kTmemCols);
    tc_relinquish();
  }
  if (tid == 0) {
    mbar_init(bar, 1);
    fence_mbar_init();
  }
  // X tile to fp16 (rows past nq are zero)
  // thread i fills row 8 (i / 8 / kx) + i % 8, chunk (i / 8) % kx: eight
  // consecutive threads write one 128-byte core matrix (no bank conflicts)
  for (int i = tid; i < kRows * kx; i += 128) {
    const int c = (i >> 3) % kx, r = ((i >> 3) / kx) * 8 + (i & 7);
    const int64_t row = row0 + r;
    __align__(16) __half hv[8];
    if (row < nq) {
      if (DT == 0) {
        const uint2 v = *reinterpret_cast<const uint2 *>(static_cast<const uint8_t *>(x) + row * D + c * 8);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          hv[e] = __uint2half_rn((v.x >> (8 * e)) & 0xffu);
          hv[4 + e] = __uint2half_rn((v.y >> (8 * e)) & 0xffu);
        }
      } else {
        const float4 *src = reinterpret_cast<const float4 *>(static_cast<const float *>(x) + row * D + c * 8);
        const float4 u = src[0], w = src[1];
        hv[0] = __float2half_rn(u.x); hv[1] = __float2half_rn(u.y);
        hv[2] = __float2half_rn(u.z); hv[3] = __float2half_rn(u.w);
        hv[4] = __float2half_rn(w.x); hv[5] = __float2half_rn(w.y);
        hv[6] = __float2half_rn(w.z); hv[7] = __float2half_rn(w.w);
      }
    } else {
#pragma unroll
      for (int e = 0; e < 8; ++e) hv[e] = __float2half_rn(0.0f);
    }
    *reinterpret_cast<uint4 *>(sX + kmajor_off(r, c, kx)) = *reinterpret_cast<const uint4 *>(hv);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t d1 = tmem, d2 = tmem + kHC;
  const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
  const int r = warp * 32 + lane;  // this thread's row = TMEM lane
  const uint32_t idesc1 = mma_idesc(kRows, kHC), idesc2 = mma_idesc(kRows, n2);
  uint32_t phase = 0;
  int ok = 1;
  for (int hc = 0; hc < H / kHC && ok; ++hc) {
    // operands of this chunk: W1 rows [hc*128, +128), W2 columns [hc*128, +128)
    for (int i = tid; i < kHC * kx; i += 128) {
      const int c = (i >> 3) % kx, n = ((i >> 3) / kx) * 8 + (i & 7);
      *reinterpret_cast<uint4 *>(sW1 + kmajor_off(n, c, kx)) =
          *reinterpret_cast<const uint4 *>(W1h + (size_t)(hc * kHC + n) * D + c * 8);
    }
    for (int i = tid; i < n2 * 16; i += 128) {
      const int c = (i >> 3) & 15, n = (i >> 7) * 8 + (i & 7);
      *reinterpret_cast<uint4 *>(sW2 + kmajor_off(n, c, 16)) =
          *reinterpret_cast<const uint4 *>(W2h + (size_t)n * H + hc * kHC + c * 8);
    }
    sb1[tid] = b1[hc * kHC + tid];
    fence_async_smem();
    tc_fence_before();
    __syncthreads();
    if (tid == 0) {
      tc_fence_after();
      for (int ks = 0; ks < D / 16; ++ks)
        tc_mma_f16(d1, smem_desc(smem_u32(sX) + ks * 256, 128, kx * 128),
                   smem_desc(smem_u32(sW1) + ks * 256, 128, kx * 128), idesc1, ks > 0 ? 1u : 0u);
      tc_commit(bar);
    }
    ok = __syncthreads_and(mbar_wait_bounded(bar, phase));
    phase ^= 1;
    if (!ok) break;
    tc_fence_after();
    // h = ReLU(s * acc + b1) -> fp16 A operand of layer 2
#pragma unroll 1
    for (int cb = 0; cb < kHC; cb += 32) {
      uint32_t v[32];
      tc_ld32(d1 + lane_base + (uint32_t)cb, v);
      tc_wait_ld();
#pragma unroll
      for (int j8 = 0; j8 < 4; ++j8) {
        __align__(16) __half hv[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const int j = cb + j8 * 8 + e;
          const float h = __fmaf_rn(s, __uint_as_float(v[j8 * 8 + e]), sb1[j]);
          hv[e] = __float2half_rn(h > 0.0f ? h : 0.0f);
        }
        *reinterpret_cast<uint4 *>(sH + kmajor_off(r, (cb >> 3) + j8, 16)) =
            *reinterpret_cast<const uint4 *>(hv);
      }
    }
    fence_async_smem();
    tc_fence_before();
    __syncthreads();
    if (tid == 0) {
      tc_fence_after();
      for (int ks = 0; ks < kHC / 16; ++ks)
        tc_mma_f16(d2, smem_desc(smem_u32(sH) + ks * 256, 128, 16 * 128),
                   smem_desc(smem_u32(sW2) + ks * 256, 128, 16 * 128), idesc2,
                   (hc > 0 || ks > 0) ? 1u : 0u);
      tc_commit(bar);
    }
    ok = __syncthreads_and(mbar_wait_bounded(bar, phase));
    phase ^= 1;
    tc_fence_after();
  }
  if (ok) {
    uint32_t v[32];
    tc_ld32(d2 + lane_base, v);
    tc_wait_ld();
    const int64_t row = row0 + r;
    if (row < nq)
      for (int j = 0; j < b; ++j) out[row * b + j] = __fadd_rn(__uint_as_float(v[j]), b2[j]);
  } else if (tid == 0) {
    atomicCAS(err, 0, NR_DEV_TIMEOUT);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tc_dealloc(tmem, kTmemCols);
  }
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
  return ix->W1h != nullptr && ix->D % 16 == 0 && ix->D <= 256 && ix->H % kHC == 0 && ix->b <= 32;
}

cudaError_t nr_launch_encode(nr_index *ix, const void *d_x, int64_t nq, float *d_logits,
                             cudaStream_t s) {
  if (nq <= 0) return cudaSuccess;
  if (nr_encode_uses_tensor_cores(ix)) {
    const int n2 = ix->b <= 16 ? 16 : 32;
    const size_t smem = (size_t)kRows * ix->D * 2 + (size_t)kHC * ix->D * 2 +
                        (size_t)kRows * kHC * 2 + (size_t)n2 * kHC * 2 + kHC * 4 + 16;
    auto kern = ix->dtype == 0 ? encode_tc_kernel<0> : encode_tc_kernel<1>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int64_t grid = (nq + kRows - 1) / kRows;
    kern<<<(unsigned)grid, 128, smem, s>>>(d_x, ix->D, ix->H, ix->b, n2, ix->in_scale,
                                           static_cast<const __half *>(ix->W1h), ix->b1,
                                           static_cast<const __half *>(ix->W2h), ix->b2, nq,
                                           d_logits, ix->d_err);
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
