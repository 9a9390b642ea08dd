// Blackwell (sm_103a) building blocks in inline PTX: mbarriers with bounded
// waits, TMA tensor loads, tensor-memory allocation / loads / stores, and
// tcgen05 MMA with shared-memory matrix descriptors (bf16 in, fp32 out).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace ltd {
namespace tc {

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t globaltimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// ------------------------------------------------------------- mbarriers
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_init_fence() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// Like mbar_try, but a thread whose phase has not completed is suspended
// in hardware until it completes or about `ns` nanoseconds have passed,
// instead of returning at once.
__device__ __forceinline__ bool mbar_try_suspend(uint32_t bar, uint32_t parity, uint32_t ns) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity), "r"(ns)
      : "memory");
  return ok != 0;
}

// Every wait gives up after this long (the caller then flags a timeout and
// winds down instead of spinning forever).
constexpr uint64_t kWaitLimitNs = 1000000000ull;

// Wait until the phase with the given parity has completed; false on timeout.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
  if (mbar_try(bar, parity)) return true;
  const uint64_t t0 = globaltimer();
  while (true) {
#pragma unroll 1
    for (int i = 0; i < 64; ++i)
      if (mbar_try(bar, parity)) return true;
    if (globaltimer() - t0 > kWaitLimitNs) return false;
  }
}
// The same wait, but between tries the thread sleeps in hardware (up to 1 us
// a try) rather than re-issuing the test, so a waiting warp takes no issue
// slots from the warps that work.  It pays where many warps wait while a few
// compute (the attention kernel: 0.06-0.1 us per 8B- and 13B-class layer);
// a pipeline that waits on every stage (the LM-head GEMM) lost 2-13% to the
// later wake-up.
__device__ __forceinline__ bool mbar_wait_sleep(uint32_t bar, uint32_t parity) {
  if (mbar_try(bar, parity)) return true;
  const uint64_t t0 = globaltimer();
  while (true) {
    if (mbar_try_suspend(bar, parity, 1000u)) return true;
    if (globaltimer() - t0 > kWaitLimitNs) return false;
  }
}

// ------------------------------------------------------------------- TMA
__device__ __forceinline__ void tma_prefetch(const CUtensorMap* map) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}
// 3-D tiled load into shared memory; completes `bytes` on mbarrier `bar`.
// The innermost coordinate c0 times the element size must be a multiple of
// 16 bytes (every caller passes 0 or 64 bf16 elements).
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* map, uint32_t bar,
                                            int32_t c0, int32_t c1, int32_t c2) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(c0), "r"(c1), "r"(c2)
      : "memory");
}

// 4-D tiled load into shared memory (same rules as the 3-D load).
__device__ __forceinline__ void tma_load_4d(uint32_t dst, const CUtensorMap* map, uint32_t bar,
                                            int32_t c0, int32_t c1, int32_t c2, int32_t c3) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4, %5, %6}], [%2];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(c0), "r"(c1), "r"(c2), "r"(c3)
      : "memory");
}

// ------------------------------------------------------- tensor memory
__device__ __forceinline__ void tmem_alloc(uint32_t holder_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(holder_smem),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void fence_before_sync() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void fence_after_sync() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// Generic-proxy shared-memory writes become visible to the tensor core.
__device__ __forceinline__ void fence_smem_async() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
// Arrive on `bar` once every MMA issued so far by this thread completes.
__device__ __forceinline__ void mma_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   bar)
               : "memory");
}

// 32 consecutive 32-bit columns of this thread's TMEM lane.
struct Frag32 {
  uint32_t r[32];
};
// Load and wait in one statement: the destination registers are written by
// the asynchronous load, so no instruction the compiler might place between
// a separate load and wait (a copy, a reuse of a register it believes
// already written) can touch them early.
__device__ __forceinline__ void tmem_ld32_sync(uint32_t taddr, Frag32& f) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(f.r[0]), "=r"(f.r[1]), "=r"(f.r[2]), "=r"(f.r[3]), "=r"(f.r[4]), "=r"(f.r[5]), "=r"(f.r[6]), "=r"(f.r[7]), "=r"(f.r[8]), "=r"(f.r[9]), "=r"(f.r[10]), "=r"(f.r[11]), "=r"(f.r[12]), "=r"(f.r[13]), "=r"(f.r[14]), "=r"(f.r[15]), "=r"(f.r[16]), "=r"(f.r[17]), "=r"(f.r[18]), "=r"(f.r[19]), "=r"(f.r[20]), "=r"(f.r[21]), "=r"(f.r[22]), "=r"(f.r[23]), "=r"(f.r[24]), "=r"(f.r[25]), "=r"(f.r[26]), "=r"(f.r[27]), "=r"(f.r[28]), "=r"(f.r[29]), "=r"(f.r[30]), "=r"(f.r[31])
      : "r"(taddr));
}
struct Frag16 {
  uint32_t r[16];
};
// A whole 128-column row per thread (32x32b.x128) and a 64-column store.
struct Frag128 {
  uint32_t r[128];
};
__device__ __forceinline__ void tmem_ld128_sync(uint32_t taddr, Frag128& f) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x128.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32, %33, %34, %35, %36, %37, %38, %39, %40, %41, %42, %43, %44, %45, %46, %47, %48, %49, %50, %51, %52, %53, %54, %55, %56, %57, %58, %59, %60, %61, %62, %63, %64, %65, %66, %67, %68, %69, %70, %71, %72, %73, %74, %75, %76, %77, %78, %79, %80, %81, %82, %83, %84, %85, %86, %87, %88, %89, %90, %91, %92, %93, %94, %95, %96, %97, %98, %99, %100, %101, %102, %103, %104, %105, %106, %107, %108, %109, %110, %111, %112, %113, %114, %115, %116, %117, %118, %119, %120, %121, %122, %123, %124, %125, %126, %127}, [%128];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(f.r[0]), "=r"(f.r[1]), "=r"(f.r[2]), "=r"(f.r[3]), "=r"(f.r[4]), "=r"(f.r[5]), "=r"(f.r[6]), "=r"(f.r[7]), "=r"(f.r[8]), "=r"(f.r[9]), "=r"(f.r[10]), "=r"(f.r[11]), "=r"(f.r[12]), "=r"(f.r[13]), "=r"(f.r[14]), "=r"(f.r[15]), "=r"(f.r[16]), "=r"(f.r[17]), "=r"(f.r[18]), "=r"(f.r[19]), "=r"(f.r[20]), "=r"(f.r[21]), "=r"(f.r[22]), "=r"(f.r[23]), "=r"(f.r[24]), "=r"(f.r[25]), "=r"(f.r[26]), "=r"(f.r[27]), "=r"(f.r[28]), "=r"(f.r[29]), "=r"(f.r[30]), "=r"(f.r[31]), "=r"(f.r[32]), "=r"(f.r[33]), "=r"(f.r[34]), "=r"(f.r[35]), "=r"(f.r[36]), "=r"(f.r[37]), "=r"(f.r[38]), "=r"(f.r[39]), "=r"(f.r[40]), "=r"(f.r[41]), "=r"(f.r[42]), "=r"(f.r[43]), "=r"(f.r[44]), "=r"(f.r[45]), "=r"(f.r[46]), "=r"(f.r[47]), "=r"(f.r[48]), "=r"(f.r[49]), "=r"(f.r[50]), "=r"(f.r[51]), "=r"(f.r[52]), "=r"(f.r[53]), "=r"(f.r[54]), "=r"(f.r[55]), "=r"(f.r[56]), "=r"(f.r[57]), "=r"(f.r[58]), "=r"(f.r[59]), "=r"(f.r[60]), "=r"(f.r[61]), "=r"(f.r[62]), "=r"(f.r[63]), "=r"(f.r[64]), "=r"(f.r[65]), "=r"(f.r[66]), "=r"(f.r[67]), "=r"(f.r[68]), "=r"(f.r[69]), "=r"(f.r[70]), "=r"(f.r[71]), "=r"(f.r[72]), "=r"(f.r[73]), "=r"(f.r[74]), "=r"(f.r[75]), "=r"(f.r[76]), "=r"(f.r[77]), "=r"(f.r[78]), "=r"(f.r[79]), "=r"(f.r[80]), "=r"(f.r[81]), "=r"(f.r[82]), "=r"(f.r[83]), "=r"(f.r[84]), "=r"(f.r[85]), "=r"(f.r[86]), "=r"(f.r[87]), "=r"(f.r[88]), "=r"(f.r[89]), "=r"(f.r[90]), "=r"(f.r[91]), "=r"(f.r[92]), "=r"(f.r[93]), "=r"(f.r[94]), "=r"(f.r[95]), "=r"(f.r[96]), "=r"(f.r[97]), "=r"(f.r[98]), "=r"(f.r[99]), "=r"(f.r[100]), "=r"(f.r[101]), "=r"(f.r[102]), "=r"(f.r[103]), "=r"(f.r[104]), "=r"(f.r[105]), "=r"(f.r[106]), "=r"(f.r[107]), "=r"(f.r[108]), "=r"(f.r[109]), "=r"(f.r[110]), "=r"(f.r[111]), "=r"(f.r[112]), "=r"(f.r[113]), "=r"(f.r[114]), "=r"(f.r[115]), "=r"(f.r[116]), "=r"(f.r[117]), "=r"(f.r[118]), "=r"(f.r[119]), "=r"(f.r[120]), "=r"(f.r[121]), "=r"(f.r[122]), "=r"(f.r[123]), "=r"(f.r[124]), "=r"(f.r[125]), "=r"(f.r[126]), "=r"(f.r[127])
      : "r"(taddr));
}
struct Frag64 {
  uint32_t r[64];
};
// 64 columns, load and wait in one statement (see tmem_ld32_sync).
__device__ __forceinline__ void tmem_ld64_sync(uint32_t taddr, Frag64& f) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x64.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32, %33, %34, %35, %36, %37, %38, %39, %40, %41, %42, %43, %44, %45, %46, %47, %48, %49, %50, %51, %52, %53, %54, %55, %56, %57, %58, %59, %60, %61, %62, %63}, [%64];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(f.r[0]), "=r"(f.r[1]), "=r"(f.r[2]), "=r"(f.r[3]), "=r"(f.r[4]), "=r"(f.r[5]), "=r"(f.r[6]), "=r"(f.r[7]), "=r"(f.r[8]), "=r"(f.r[9]), "=r"(f.r[10]), "=r"(f.r[11]), "=r"(f.r[12]), "=r"(f.r[13]), "=r"(f.r[14]), "=r"(f.r[15]), "=r"(f.r[16]), "=r"(f.r[17]), "=r"(f.r[18]), "=r"(f.r[19]), "=r"(f.r[20]), "=r"(f.r[21]), "=r"(f.r[22]), "=r"(f.r[23]), "=r"(f.r[24]), "=r"(f.r[25]), "=r"(f.r[26]), "=r"(f.r[27]), "=r"(f.r[28]), "=r"(f.r[29]), "=r"(f.r[30]), "=r"(f.r[31]), "=r"(f.r[32]), "=r"(f.r[33]), "=r"(f.r[34]), "=r"(f.r[35]), "=r"(f.r[36]), "=r"(f.r[37]), "=r"(f.r[38]), "=r"(f.r[39]), "=r"(f.r[40]), "=r"(f.r[41]), "=r"(f.r[42]), "=r"(f.r[43]), "=r"(f.r[44]), "=r"(f.r[45]), "=r"(f.r[46]), "=r"(f.r[47]), "=r"(f.r[48]), "=r"(f.r[49]), "=r"(f.r[50]), "=r"(f.r[51]), "=r"(f.r[52]), "=r"(f.r[53]), "=r"(f.r[54]), "=r"(f.r[55]), "=r"(f.r[56]), "=r"(f.r[57]), "=r"(f.r[58]), "=r"(f.r[59]), "=r"(f.r[60]), "=r"(f.r[61]), "=r"(f.r[62]), "=r"(f.r[63])
      : "r"(taddr));
}
// Store and wait in one statement: the source registers stay untouched until
// the store has completed, whatever the compiler schedules after it.
__device__ __forceinline__ void tmem_st16_sync(uint32_t taddr, const Frag16& f) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};\n\t"
      "tcgen05.wait::st.sync.aligned;" ::"r"(taddr), "r"(f.r[0]), "r"(f.r[1]), "r"(f.r[2]), "r"(f.r[3]), "r"(f.r[4]), "r"(f.r[5]), "r"(f.r[6]), "r"(f.r[7]), "r"(f.r[8]), "r"(f.r[9]), "r"(f.r[10]), "r"(f.r[11]), "r"(f.r[12]), "r"(f.r[13]), "r"(f.r[14]), "r"(f.r[15])
      : "memory");
}
__device__ __forceinline__ void tmem_st32_sync(uint32_t taddr, const Frag32& f) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};\n\t"
      "tcgen05.wait::st.sync.aligned;" ::"r"(taddr), "r"(f.r[0]), "r"(f.r[1]), "r"(f.r[2]), "r"(f.r[3]), "r"(f.r[4]), "r"(f.r[5]), "r"(f.r[6]), "r"(f.r[7]), "r"(f.r[8]), "r"(f.r[9]), "r"(f.r[10]), "r"(f.r[11]), "r"(f.r[12]), "r"(f.r[13]), "r"(f.r[14]), "r"(f.r[15]), "r"(f.r[16]), "r"(f.r[17]), "r"(f.r[18]), "r"(f.r[19]), "r"(f.r[20]), "r"(f.r[21]), "r"(f.r[22]), "r"(f.r[23]), "r"(f.r[24]), "r"(f.r[25]), "r"(f.r[26]), "r"(f.r[27]), "r"(f.r[28]), "r"(f.r[29]), "r"(f.r[30]), "r"(f.r[31])
      : "memory");
}
// The first 64 registers of a 128-register fragment.
__device__ __forceinline__ void tmem_st64_lo_sync(uint32_t taddr, const Frag128& f) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x64.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32, %33, %34, %35, %36, %37, %38, %39, %40, %41, %42, %43, %44, %45, %46, %47, %48, %49, %50, %51, %52, %53, %54, %55, %56, %57, %58, %59, %60, %61, %62, %63, %64};\n\t"
      "tcgen05.wait::st.sync.aligned;" ::"r"(taddr), "r"(f.r[0]), "r"(f.r[1]), "r"(f.r[2]), "r"(f.r[3]), "r"(f.r[4]), "r"(f.r[5]), "r"(f.r[6]), "r"(f.r[7]), "r"(f.r[8]), "r"(f.r[9]), "r"(f.r[10]), "r"(f.r[11]), "r"(f.r[12]), "r"(f.r[13]), "r"(f.r[14]), "r"(f.r[15]), "r"(f.r[16]), "r"(f.r[17]), "r"(f.r[18]), "r"(f.r[19]), "r"(f.r[20]), "r"(f.r[21]), "r"(f.r[22]), "r"(f.r[23]), "r"(f.r[24]), "r"(f.r[25]), "r"(f.r[26]), "r"(f.r[27]), "r"(f.r[28]), "r"(f.r[29]), "r"(f.r[30]), "r"(f.r[31]), "r"(f.r[32]), "r"(f.r[33]), "r"(f.r[34]), "r"(f.r[35]), "r"(f.r[36]), "r"(f.r[37]), "r"(f.r[38]), "r"(f.r[39]), "r"(f.r[40]), "r"(f.r[41]), "r"(f.r[42]), "r"(f.r[43]), "r"(f.r[44]), "r"(f.r[45]), "r"(f.r[46]), "r"(f.r[47]), "r"(f.r[48]), "r"(f.r[49]), "r"(f.r[50]), "r"(f.r[51]), "r"(f.r[52]), "r"(f.r[53]), "r"(f.r[54]), "r"(f.r[55]), "r"(f.r[56]), "r"(f.r[57]), "r"(f.r[58]), "r"(f.r[59]), "r"(f.r[60]), "r"(f.r[61]), "r"(f.r[62]), "r"(f.r[63])
      : "memory");
}
__device__ __forceinline__ void tmem_wait_st() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// ------------------------------------------------------- MMA descriptors
// Shared-memory matrix descriptor, 128-byte swizzle (tcgen05 format):
// start address >> 4 in bits 0-13, leading-dimension byte offset >> 4 in
// 16-29, stride-dimension byte offset >> 4 in 32-45, the fixed 0b001 in
// 46-48, base offset 0 (atoms are 1024-byte aligned), swizzle mode 2 (128B)
// in 61-63.  K-major operands: SBO = 1024 (eight 128-byte rows), LBO unused.
// MN-major operands: LBO = bytes between 64-element MN blocks, SBO = bytes
// between groups of eight K rows.
__device__ __forceinline__ uint64_t sdesc_sw128(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  return static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4) |
         (static_cast<uint64_t>((lbo >> 4) & 0x3FFFu) << 16) |
         (static_cast<uint64_t>((sbo >> 4) & 0x3FFFu) << 32) | (1ull << 46) | (2ull << 61);
}

// Instruction descriptor of kind::f16 with bf16 A/B and fp32 accumulation:
// D format (bits 4-5) = F32, A and B formats (7-9, 10-12) = BF16, A K-major,
// B K-major or MN-major (bit 16), N >> 3 in bits 17-22, M >> 4 in 24-28.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N, bool b_mn_major) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((b_mn_major ? 1u : 0u) << 16) |
         (static_cast<uint32_t>(N >> 3) << 17) | (static_cast<uint32_t>(M >> 4) << 24);
}

// D[tmem] (+)= A[smem] * B[smem], one elected thread issues it.
__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                         uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// D[tmem] (+)= A[tmem] * B[smem]: A (M x K, 16-bit, two K elements per
// 32-bit column, row i in lane i) is read from tensor memory.
__device__ __forceinline__ void mma_bf16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc,
                                            uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// ------------------------------------------------- thread-block clusters
// (a kernel launched without a cluster is a cluster of one CTA)
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// Every thread of every CTA in the cluster must call this.
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\t"
               "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// Address of the same shared-memory location in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t mapa(uint32_t saddr, uint32_t rank) {
  uint32_t r;
  asm("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
  return r;
}
__device__ __forceinline__ uint64_t ld_cluster_u64(uint32_t caddr) {
  uint64_t v;
  asm volatile("ld.shared::cluster.u64 %0, [%1];" : "=l"(v) : "r"(caddr) : "memory");
  return v;
}
// Named barrier `id` over `nthreads` threads (whole warps) that also returns
// the AND of `p` over them.
__device__ __forceinline__ bool bar_red_and(int id, int nthreads, bool p) {
  int r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\tsetp.ne.b32 p, %1, 0;\n\t"
      "bar.red.and.pred q, %2, %3, p;\n\tselp.b32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"(static_cast<int>(p)), "r"(id), "r"(nthreads)
      : "memory");
  return r != 0;
}
// Three-input maximum (sm_100 and later).
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}
__device__ __forceinline__ uint32_t ld_acquire_gpu(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void red_add_release_gpu(uint32_t* p, uint32_t v) {
  asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ void st_cluster_f1(uint32_t caddr, float v) {
  asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(caddr), "f"(v) : "memory");
}
__device__ __forceinline__ void bulk_commit() {
  asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}
// Bulk (untiled) copies: 16-byte aligned addresses, sizes a multiple of 16.
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
      "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}
__device__ __forceinline__ void bulk_s2g(void* dst, uint32_t src, uint32_t bytes) {
  asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst), "r"(src),
               "r"(bytes)
               : "memory");
}
// Ask L2 to fetch `bytes` (a multiple of 16) from global memory at `p`.
__device__ __forceinline__ void prefetch_l2(const void* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}
// Wait until this thread's bulk copies have completed (writes performed).
__device__ __forceinline__ void bulk_wait_all() {
  asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}
__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

}  // namespace tc

// Host: encode a 3-D bf16 tensor map with 128-byte swizzle (dims innermost
// first, strides in bytes for dims 1 and 2).  Returns false on failure.
bool encode_tmap_bf16_3d(CUtensorMap* map, const void* base, uint64_t d0, uint64_t d1, uint64_t d2,
                         uint64_t stride1, uint64_t stride2, uint32_t b0, uint32_t b1, uint32_t b2);

}  // namespace ltd
