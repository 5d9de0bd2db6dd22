// 5th-generation tensor core (tcgen05) helpers: TMEM allocation, UMMA
// issue/commit, TMEM loads, shared-memory matrix descriptors, TMA gather4 and
// vector reductions.  Inline PTX for sm_100-family (built for sm_103a).
//
// Conventions used by the GEMM kernels:
//  * D[128 x N] (fp32, TMEM lanes 0..127 = rows, columns 0..N-1) +=
//    A[128 x K] * B[N x K]^T, both bf16 and K-major ("row-major with K
//    contiguous"), staged in shared memory by TMA with the 128-byte swizzle:
//    a tile row is 64 bf16 (128 B), 8-row groups are 1024 B apart.
//  * One UMMA instruction covers K = 16; the four K = 16 slices of a 64-wide
//    tile are addressed by advancing the descriptor start address 32 B.
#pragma once

#include "pp_common.cuh"

namespace pp {

// ------------------------------------------------------------------- TMEM
PP_DEVINL void tmem_alloc(uint32_t* dst_smem, uint32_t ncols) {  // whole warp
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(dst_smem)),
                 "r"(ncols)
                 : "memory");
}
PP_DEVINL void tmem_relinquish() {  // whole warp
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
PP_DEVINL void tmem_dealloc(uint32_t taddr, uint32_t ncols) {  // whole warp
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
PP_DEVINL void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
PP_DEVINL void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// --------------------------------------------------------------- UMMA issue
// Instruction descriptor, kind::f16: D fp32, A and B bf16, both K-major,
// M = 128, N (multiple of 16, 16..256).
PP_DEVINL constexpr uint32_t idesc_bf16_m128(int n) {
    return (1u << 4)                      // D format: f32
           | (1u << 7)                    // A format: bf16
           | (1u << 10)                   // B format: bf16
           | ((uint32_t)(n >> 3) << 17)   // N >> 3
           | ((uint32_t)(128 >> 4) << 24);  // M >> 4
}

// Shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row groups
// 1024 B apart.  `p` must lie in a 1024-byte aligned tile (plus a multiple
// of 32 B to select a K = 16 slice).
PP_DEVINL uint64_t sdesc_sw128(const void* p) {
    const uint32_t a = smem_u32(p);
    uint64_t d = (uint64_t)((a & 0x3ffffu) >> 4);  // start address
    d |= (uint64_t)1u << 16;                         // leading byte offset (unused by SW128 K-major)
    d |= (uint64_t)(1024u >> 4) << 32;               // stride byte offset: 8 rows x 128 B
    d |= (uint64_t)1u << 46;                         // descriptor version
    d |= (uint64_t)2u << 61;                         // 128-byte swizzle
    return d;
}

PP_DEVINL void umma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Arrive on `bar` once every previously issued UMMA of this thread is done.
PP_DEVINL void umma_commit(uint64_t* bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                     smem_u32(bar))
                 : "memory");
}

// D[128 x N] (+)= A_tile[128 x 64] * B_tile[N x 64]^T : four K = 16 UMMAs.
PP_DEVINL void umma_k64(uint32_t d_tmem, const void* a_tile, const void* b_tile, uint32_t idesc, bool accumulate) {
    const uint64_t ad = sdesc_sw128(a_tile), bd = sdesc_sw128(b_tile);
#pragma unroll
    for (int k = 0; k < 4; k++)
        umma_bf16(d_tmem, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), idesc, (accumulate || k > 0) ? 1u : 0u);
}

// ------------------------------------------------------------ TMEM -> regs
// Warp-collective: lane i receives row (lane base + i), 32 consecutive
// fp32 columns starting at the address's column.
PP_DEVINL void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, "
        "%14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
}
// Same with 16 columns.
PP_DEVINL void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, "
        "%14, %15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
}
PP_DEVINL void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// --------------------------------------------------------------- TMA extra
// Four rows (row0..row3) of a 2-D tensor, one box of {64 x 1} each, landing
// as four consecutive 128-byte rows at dst (the tensor map's box is one row
// high).  col * 2 B must be a multiple of 16 B.
PP_DEVINL void tma_gather4(void* dst, const CUtensorMap* map, int col, int r0, int r1, int r2, int r3,
                           uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile::gather4.mbarrier::complete_tx::bytes [%0], [%1, "
        "{%2, %3, %4, %5, %6}], [%7];" ::"r"(smem_u32(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(col), "r"(r0), "r"(r1), "r"(r2), "r"(r3), "r"(smem_u32(bar))
        : "memory");
}

// 16-byte cp.async global -> shared through L2 (not L1); src_bytes = 0
// writes 16 zero bytes instead of reading.  Completion: cp_async_commit
// closes a group, cp_async_wait<N> waits until at most N groups are pending.
PP_DEVINL void cp_async_16(void* dst, const void* src, uint32_t src_bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(dst)), "l"(src), "r"(src_bytes)
                 : "memory");
}

PP_DEVINL void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }

template <int N>
PP_DEVINL void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// 2-D tiled store shared -> global of one box (c0, c1 >= 0; the part of the
// box past the tensor's extent is not written), tracked as a bulk group of
// the issuing thread.
PP_DEVINL void tma_store_2d(const CUtensorMap* map, const void* src, int c0, int c1) {
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.tile.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
                     reinterpret_cast<uint64_t>(map)),
                 "r"(smem_u32(src)), "r"(c0), "r"(c1)
                 : "memory");
}

PP_DEVINL void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// the shared-memory sources of all but the N most recent committed bulk
// groups have been read
template <int N>
PP_DEVINL void bulk_wait_read() {
    asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}
// all committed bulk groups are complete (their global writes done)
PP_DEVINL void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// y[0..3] += v (fp32, one 16-byte vector reduction in L2)
PP_DEVINL void red_add_v4(float* addr, float a, float b, float c, float d) {
    asm volatile("red.global.add.v4.f32 [%0], {%1, %2, %3, %4};" ::"l"(addr), "f"(a), "f"(b), "f"(c), "f"(d)
                 : "memory");
}

PP_DEVINL uint32_t pack_bf16x2(float lo, float hi) {
    const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t*>(&v);
}

}  // namespace pp
