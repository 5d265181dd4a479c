// Blackwell 5th-generation tensor cores (tcgen05) for the prefill scoring contraction: operands
// in shared memory as K-major tiles with the 128-byte swizzle, the fp32 accumulator in tensor
// memory (TMEM), the MMA issued by one thread and its completion signalled on an mbarrier.
#pragma once

#include <cuda_fp16.h>
#include <stdint.h>

#include "mkv_common.cuh"

namespace mkv {

// Operand tile layout (K-major, 128-byte swizzle, as TMA writes it with the 128-byte swizzle mode
// into a 1024-byte aligned destination): a row's K extent is cut into atoms of 64 fp16 (128 B); an
// atom of R rows is R * 128 B, rows in 8-row groups of 1024 B, and the 16-byte chunk c of row r sits
// at chunk c ^ (r % 8).

// Shared-memory matrix descriptor of such a tile starting at shared address `start`: start >> 4 in
// bits [0,14), leading byte offset >> 4 in [16,30) (unused by swizzled K-major tiles), stride byte
// offset >> 4 in [32,46) (1024 B between 8-row groups), descriptor version 1 in [46,48), layout
// 128-byte swizzle (2) in [61,64).  A K step of 16 elements advances `start` by 32 bytes.
__device__ __forceinline__ uint64_t tc_desc_sw128(uint32_t start) {
  uint64_t d = 0;
  d |= (uint64_t)((start >> 4) & 0x3fffu);
  d |= (uint64_t)1u << 16;
  d |= (uint64_t)(1024u >> 4) << 32;
  d |= (uint64_t)1u << 46;
  d |= (uint64_t)2u << 61;
  return d;
}

// Instruction descriptor of kind::f16 with an fp32 accumulator, A and B fp16 and K-major:
// D format f32 in bits [4,6), N >> 3 in [17,23), M >> 4 in [24,29).
__host__ __device__ constexpr uint32_t tc_idesc_f16(int M, int N) {
  return (1u << 4) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ void tc_mbar_init(uint64_t* bar, int count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}
// One test of phase `parity` of `bar` (true once that phase has completed)
__device__ __forceinline__ bool tc_mbar_try(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2; selp.u32 %0, 1, 0, p; }"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
// The GPU's global nanosecond clock
__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
// Bounded wait on phase `parity` of `bar`: false if it has not completed within `ns` nanoseconds.
__device__ __forceinline__ bool tc_mbar_wait(uint64_t* bar, uint32_t parity, uint64_t ns) {
  if (tc_mbar_try(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  while (!tc_mbar_try(bar, parity))
    if (globaltimer_ns() - t0 > ns) return false;
  return true;
}
__device__ __forceinline__ void tc_mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}
// arrive on `bar` and add `bytes` to the transaction count its current phase waits for
__device__ __forceinline__ void tc_mbar_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
               : "memory");
}
// TMA: the box at coordinates (x, y, z, w) of the tensor map at generic address `map` into shared
// memory at `dst`, completing its bytes of `bar`'s transaction count (x * element size must be a
// multiple of 16 bytes; rows outside the tensor are zero-filled)
__device__ __forceinline__ void tma_load_4d(void* dst, const void* map, int x, int y, int z, int w, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4, %5}], [%6];" ::
          "r"(smem_addr(dst)),
      "l"(map), "r"(x), "r"(y), "r"(z), "r"(w), "r"(smem_addr(bar))
      : "memory");
}
// bulk copy of `bytes` (a multiple of 16; both addresses 16-byte aligned) into shared memory
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   smem_addr(dst)),
               "l"(src), "r"(bytes), "r"(smem_addr(bar))
               : "memory");
}
// TMEM columns (a power of two >= 32) for this CTA, the base address written to `*dst` (one warp)
__device__ __forceinline__ void tc_alloc(uint32_t* dst, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_addr(dst)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tc_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
// D[tmem] (+)= A[smem] B[smem]^T, fp16 in, fp32 accumulate; `acc` 0 overwrites D
__device__ __forceinline__ void tc_mma(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
  asm volatile("{ .reg .pred p; setp.ne.b32 p, %4, 0;\n tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p; }"
               ::"r"(d_tmem), "l"(a), "l"(b), "r"(idesc), "r"(acc)
               : "memory");
}
// arrive on `bar` once every MMA this thread issued so far has completed
__device__ __forceinline__ void tc_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   smem_addr(bar))
               : "memory");
}
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
// 32 TMEM lanes x 16 consecutive fp32 columns: thread i of the warp gets lane (address lane + i).
// The registers are valid only after a tcgen05.wait::ld (tc_wait_ld_regs).
__device__ __forceinline__ void tc_ld16_issue(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}
// Wait for this thread's tensor-memory loads.  The wait names the 32 loaded registers of r, so
// the compiler orders every use of them after it (a second wait, already satisfied, covers more).
__device__ __forceinline__ void tc_wait_ld_regs(uint32_t (&r)[32]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]),
                 "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]),
                 "+r"(r[15]), "+r"(r[16]), "+r"(r[17]), "+r"(r[18]), "+r"(r[19]), "+r"(r[20]), "+r"(r[21]),
                 "+r"(r[22]), "+r"(r[23]), "+r"(r[24]), "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]),
                 "+r"(r[29]), "+r"(r[30]), "+r"(r[31])
               :
               : "memory");
}

// 64 consecutive fp32 columns (four loads in flight, then the wait)
__device__ __forceinline__ void tc_ld64(uint32_t taddr, float (&v)[64]) {
  uint32_t r0[32], r1[32];
  tc_ld16_issue(taddr, *reinterpret_cast<uint32_t(*)[16]>(&r0[0]));
  tc_ld16_issue(taddr + 16, *reinterpret_cast<uint32_t(*)[16]>(&r0[16]));
  tc_ld16_issue(taddr + 32, *reinterpret_cast<uint32_t(*)[16]>(&r1[0]));
  tc_ld16_issue(taddr + 48, *reinterpret_cast<uint32_t(*)[16]>(&r1[16]));
  tc_wait_ld_regs(r0);
  tc_wait_ld_regs(r1);
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    v[i] = __uint_as_float(r0[i]);
    v[32 + i] = __uint_as_float(r1[i]);
  }
}

// Packed fp32 pairs (Blackwell): each lane of fma.rn.f32x2 / add.rn.f32x2 rounds as its scalar form
__device__ __forceinline__ uint64_t pk2(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ float2 upk2(uint64_t x) {
  float2 r;
  asm("mov.b64 {%0, %1}, %2;" : "=f"(r.x), "=f"(r.y) : "l"(x));
  return r;
}
__device__ __forceinline__ uint64_t ffma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t fadd2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
// max of three (one instruction)
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// 2^x by the special-function unit's approximation (one instruction; results below the normal
// range flush to zero, 2^-inf = 0)
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

}  // namespace mkv
