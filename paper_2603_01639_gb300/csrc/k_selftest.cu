// Diagnostic: one 128x128x128 bf16 GEMM through the same TMA -> shared memory
// -> tcgen05.mma -> tensor memory -> registers path the tree-attention kernel
// uses, for both operand layouts it needs:
//   mode 0: C = A * B^T, B stored [N][K] (K-major, like S = Q K^T)
//   mode 1: C = A * B,   B stored [K][N] (MN-major, like O = P V)
// A, B are row-major bf16 [128][128]; C is row-major fp32 [128][128].
#include "ltd_common.cuh"
#include "ltd_internal.h"
#include "tc_util.cuh"

namespace ltd {

namespace {

constexpr uint32_t kHalf = 16384;

__global__ void __launch_bounds__(128) umma_selftest_kernel(const __grid_constant__ CUtensorMap ta,
                                                            const __grid_constant__ CUtensorMap tb,
                                                            float* __restrict__ C, int mode,
                                                            uint32_t* err) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = tc::smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  const uint32_t sA = base, sB = base + 2 * kHalf;
  const uint32_t bar_load = base + 4 * kHalf, bar_mma = bar_load + 8;
  uint32_t* holder = reinterpret_cast<uint32_t*>(gbase + 4 * kHalf + 16);
  const int tid = threadIdx.x, warp = tid >> 5;

  if (tid == 0) {
    tc::mbar_init(bar_load, 1);
    tc::mbar_init(bar_mma, 1);
    tc::mbar_init_fence();
  }
  if (warp == 0) {
    tc::tmem_alloc(tc::smem_u32(holder), 128);
    tc::tmem_relinquish();
  }
  tc::fence_before_sync();
  __syncthreads();
  tc::fence_after_sync();
  const uint32_t tmem = *holder;

  if (tid == 0) {
    tc::tma_prefetch(&ta);
    tc::tma_prefetch(&tb);
    tc::mbar_expect_tx(bar_load, 4 * kHalf);
    for (int h = 0; h < 2; ++h) {
      tc::tma_load_3d(sA + h * kHalf, &ta, bar_load, h * 64, 0, 0);
      tc::tma_load_3d(sB + h * kHalf, &tb, bar_load, h * 64, 0, 0);
    }
    if (tc::mbar_wait(bar_load, 0)) {
      tc::fence_after_sync();
      const uint32_t idesc = tc::idesc_bf16(128, 128, mode == 1);
      for (int ks = 0; ks < 8; ++ks) {
        const uint64_t a = tc::sdesc_sw128(sA + (ks >> 2) * kHalf + (ks & 3) * 32, 16, 1024);
        const uint64_t b = (mode == 0)
                               ? tc::sdesc_sw128(sB + (ks >> 2) * kHalf + (ks & 3) * 32, 16, 1024)
                               : tc::sdesc_sw128(sB + ks * 2048, kHalf, 1024);
        tc::mma_bf16(tmem, a, b, idesc, ks > 0 ? 1u : 0u);
      }
      tc::mma_commit(bar_mma);
    } else {
      flag_error(err, LTD_DEVERR_TIMEOUT);
    }
  }
  const bool ok = tc::mbar_wait(bar_mma, 0);
  if (!ok && tid == 0) flag_error(err, LTD_DEVERR_TIMEOUT);
  __syncwarp();
  tc::fence_after_sync();
  const int row = tid;
  for (int q = 0; q < 4; ++q) {
    tc::Frag32 f;
    tc::tmem_ld32_sync(tmem + ((32u * warp) << 16) + 32u * q, f);
    for (int j = 0; j < 32; ++j) C[row * 128 + 32 * q + j] = ok ? __uint_as_float(f.r[j]) : 0.f;
  }
  tc::fence_before_sync();
  __syncthreads();
  if (warp == 0) {
    __syncwarp();
    tc::tmem_dealloc(tmem, 128);
  }
}

}  // namespace

cudaError_t launch_umma_selftest(int mode, const void* a, const void* b, float* c, uint32_t* err,
                                 cudaStream_t s) {
  CUtensorMap ta, tb;
  if (!encode_tmap_bf16_3d(&ta, a, 128, 128, 1, 256, 256 * 128, 64, 128, 1))
    return cudaErrorInvalidValue;
  if (!encode_tmap_bf16_3d(&tb, b, 128, 128, 1, 256, 256 * 128, 64, 128, 1))
    return cudaErrorInvalidValue;
  const int smem = 4 * kHalf + 1024 + 64;
  cudaError_t e =
      cudaFuncSetAttribute(umma_selftest_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  umma_selftest_kernel<<<1, 128, smem, s>>>(ta, tb, c, mode, err);
  return cudaGetLastError();
}

}  // namespace ltd
