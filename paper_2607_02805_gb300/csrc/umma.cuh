// umma.cuh -- the 5th-generation tensor-core (tcgen05) pieces used by the SSD
// kernels: shared-memory matrix descriptors, the instruction descriptor of
// kind::f16 (bf16 operands, fp32 accumulator in TMEM), MMA issue and commit,
// mbarrier waits with an iteration limit, and 32-column TMEM loads.
//
// Operand tiles live in shared memory in the 128-byte swizzled layout: a tile
// is a set of "atoms" of 8 rows x 128 bytes (1024 bytes, 1024-byte aligned);
// inside an atom the 16-byte chunk j of row r sits at chunk (j ^ (r & 7)).
//  * K-major operand (rows are M or N, 64 bf16 of K per atom row): an atom
//    column holds all rows for 64 consecutive K, row r at byte r * 128; the
//    8-row groups are 1024 bytes apart (stride byte offset). A K step of 16
//    elements inside the atom column advances the start address by 32 bytes.
//  * MN-major operand (rows are K, 64 bf16 of N per row): the tile of N = 64
//    is one atom column, K row k at byte k * 128; 8-row K groups are 1024
//    bytes apart, so a K step of 16 advances the start address by 2048 bytes.
#pragma once
#include <cstdint>

namespace bds {
namespace umma {

// Byte offset of 16-byte chunk `chunk` of row `row` inside a swizzled region
// whose rows are 128 bytes (rows of consecutive atoms are contiguous).
__host__ __device__ constexpr uint32_t sw128(uint32_t row, uint32_t chunk) {
  return row * 128u + ((chunk ^ (row & 7u)) << 4);
}

// Shared-memory matrix descriptor, 128-byte swizzle. Fields: start address
// >> 4 (bits 0-13), leading byte offset >> 4 (16-29), stride byte offset >> 4
// (32-45), descriptor version 1 (46-47), base offset 0 (49-51), layout type 2
// = 128-byte swizzle (61-63). The leading offset is the distance between atom
// columns along M/N of an MN-major operand (unused when M/N is one atom wide)
// and is ignored for swizzled K-major operands.
__host__ __device__ constexpr uint64_t sdesc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  return (uint64_t)((saddr >> 4) & 0x3FFFu) | ((uint64_t)((lbo >> 4) & 0x3FFFu) << 16) |
         ((uint64_t)((sbo >> 4) & 0x3FFFu) << 32) | ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

// The descriptor d with its start address advanced by `bytes` (a multiple of
// 16; the advanced address stays below 256 KB, so the 14-bit field does not
// carry): one add in the MMA issue loops instead of rebuilding every field.
__host__ __device__ constexpr uint64_t sdesc_adv(uint64_t d, uint32_t bytes) { return d + (uint64_t)(bytes >> 4); }

// Instruction descriptor of tcgen05.mma kind::f16: fp32 accumulator (bits
// 4-5 = 1), bf16 A and B (7-9 = 1, 10-12 = 1), A/B major (15, 16: 0 = K-major,
// 1 = MN-major), N >> 3 (17-22), M >> 4 (24-28).
__host__ __device__ constexpr uint32_t idesc_bf16(uint32_t M, uint32_t N, bool a_mn, bool b_mn) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((a_mn ? 1u : 0u) << 15) | ((b_mn ? 1u : 0u) << 16) |
         ((N >> 3) << 17) | ((M >> 4) << 24);
}

#if defined(__CUDACC__)
__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

// D[tmem] (+)= A * B^T for one K step; issued by one thread.
__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc, bool acc) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(a), "l"(b), "r"(idesc), "r"(acc ? 1u : 0u)
      : "memory");
}

// The mbarrier at `bar` completes one phase when every MMA this thread issued
// before the commit has finished (its shared-memory reads and TMEM writes).
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(
                   smem_u32(bar))
               : "memory");
}

__device__ __forceinline__ void bar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;\n" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

// Waits for the phase with parity `parity` of `bar` to complete, at most
// `limit` polls. Returns false if it gave up.
__device__ __forceinline__ bool bar_wait(uint64_t* bar, uint32_t parity, uint32_t limit = (1u << 22)) {
  const uint32_t a = smem_u32(bar);
  for (uint32_t i = 0; i < limit; ++i) {
    uint32_t done;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(done)
        : "r"(a), "r"(parity)
        : "memory");
    if (done) return true;
  }
  return false;
}

// Generic-proxy shared-memory writes (st.shared, cp.async) made visible to
// the tensor core (async proxy); each writing thread executes it before the
// barrier that precedes the MMA issue.
__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory"); }
__device__ __forceinline__ void fence_after_sync() { asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory"); }
__device__ __forceinline__ void fence_before_sync() { asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory"); }

// 32 consecutive fp32 columns of this thread's TMEM lane (warp w reads lanes
// 32w..32w+31; `ta` carries the warp's lane base in bits 16-31).
// 32 consecutive fp32 columns of this thread's TMEM lane, without the wait:
// the registers are ready after tmem_ld_wait (on one of the loads issued
// since the last wait) and tmem_ld_after (on each of the others).
__device__ __forceinline__ void tmem_ld32_issue(uint32_t ta, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, "
      "%14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(ta));
}
// Waits for every TMEM load this thread issued; r's registers are used only after it.
__device__ __forceinline__ void tmem_ld_wait(uint32_t (&r)[32]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;\n"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]),
                 "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]),
                 "+r"(r[15]), "+r"(r[16]), "+r"(r[17]), "+r"(r[18]), "+r"(r[19]), "+r"(r[20]), "+r"(r[21]),
                 "+r"(r[22]), "+r"(r[23]), "+r"(r[24]), "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]),
                 "+r"(r[29]), "+r"(r[30]), "+r"(r[31])
               :);
}
// No instruction: orders the uses of r after the preceding tmem_ld_wait
// (volatile statements keep their order), for a second load of the same wait.
__device__ __forceinline__ void tmem_ld_after(uint32_t (&r)[32]) {
  asm volatile(""
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]),
                 "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]),
                 "+r"(r[15]), "+r"(r[16]), "+r"(r[17]), "+r"(r[18]), "+r"(r[19]), "+r"(r[20]), "+r"(r[21]),
                 "+r"(r[22]), "+r"(r[23]), "+r"(r[24]), "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]),
                 "+r"(r[29]), "+r"(r[30]), "+r"(r[31])
               :);
}
__device__ __forceinline__ void tmem_ld32(uint32_t ta, float (&v)[32]) {
  uint32_t r[32];
  tmem_ld32_issue(ta, r);
  tmem_ld_wait(r);
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}
// Two loads under one wait.
__device__ __forceinline__ void tmem_ld32x2(uint32_t ta, float (&v)[32], uint32_t tb, float (&u)[32]) {
  uint32_t r[32], q[32];
  tmem_ld32_issue(ta, r);
  tmem_ld32_issue(tb, q);
  tmem_ld_wait(r);
  tmem_ld_after(q);
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    v[i] = __uint_as_float(r[i]);
    u[i] = __uint_as_float(q[i]);
  }
}
#endif  // __CUDACC__

}  // namespace umma
}  // namespace bds
