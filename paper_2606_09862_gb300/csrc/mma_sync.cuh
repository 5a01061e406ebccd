// mma_sync.cuh -- warp-level bf16 tensor-core MMAs (m16n8k16, fp32 accumulation) on operand tiles
// kept in shared memory in the 128-byte-swizzled layout, for the chunked kernels of the decayed
// form (decay_chunk.cu).
#pragma once

#include "tc.cuh"

namespace bla {
namespace wmma16 {

// 16-byte row segments of a bf16 tile kept in the 128-byte-swizzled layout: rows of 64 elements,
// the 16-byte chunk index XOR (row & 7); columns beyond 64 in further [rows][64] blocks.
__device__ __forceinline__ uint32_t sw_off(int rows, int r, int c) {
    return (uint32_t)((c >> 6) * rows * 128 + r * 128 + ((((c & 63) >> 3) ^ (r & 7)) << 4) + (c & 7) * 2);
}

__device__ __forceinline__ void ldsm4(uint32_t addr, uint32_t (&r)[4]) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]) : "r"(addr));
}
__device__ __forceinline__ void ldsm4t(uint32_t addr, uint32_t (&r)[4]) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]) : "r"(addr));
}

// c (16x8, fp32) += a (16x16, row) * b (16x8, col)
__device__ __forceinline__ void mma16816(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
                 "{%8, %9}, {%0, %1, %2, %3};"
                 : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
                 : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// A fragment of rows [m0, m0+16) x columns [k0, k0+16) of a swizzled row-major tile.
__device__ __forceinline__ void load_a(uint32_t base, int rows, int m0, int k0, uint32_t (&a)[4]) {
    const int lane = threadIdx.x & 31;
    ldsm4(base + sw_off(rows, m0 + (lane & 15), k0 + ((lane >> 4) << 3)), a);
}
// B fragments of two 8-column tiles n0.. n0+15, k0.. k0+15, from a tile stored [n][k] (K contiguous):
// b[0], b[1] for columns n0..n0+7, b[2], b[3] for n0+8..n0+15.
__device__ __forceinline__ void load_b_nk(uint32_t base, int rows, int n0, int k0, uint32_t (&b)[4]) {
    const int lane = threadIdx.x & 31;
    ldsm4(base + sw_off(rows, n0 + (lane & 7) + ((lane >> 4) << 3), k0 + (((lane >> 3) & 1) << 3)), b);
}
// The same from a tile stored [k][n] (N contiguous), through the transposing load.
__device__ __forceinline__ void load_b_kn(uint32_t base, int rows, int n0, int k0, uint32_t (&b)[4]) {
    const int lane = threadIdx.x & 31;
    ldsm4t(base + sw_off(rows, k0 + (lane & 7) + (((lane >> 3) & 1) << 3), n0 + ((lane >> 4) << 3)), b);
}

// One 16x16 output block (two 16x8 tiles) of A [m0.., K] times B, accumulated into acc[2][4].
// B_NK: B stored [n][k]; else [k][n].
template <bool B_NK>
__device__ __forceinline__ void mma_block(uint32_t a_base, int a_rows, uint32_t b_base, int b_rows, int m0, int n0,
                                          int K, float (&acc)[2][4]) {
    for (int k0 = 0; k0 < K; k0 += 16) {
        uint32_t a[4], b[4];
        load_a(a_base, a_rows, m0, k0, a);
        if (B_NK) load_b_nk(b_base, b_rows, n0, k0, b);
        else load_b_kn(b_base, b_rows, n0, k0, b);
        mma16816(acc[0], a, b[0], b[1]);
        mma16816(acc[1], a, b[2], b[3]);
    }
}

__device__ __forceinline__ void st_bf16x2(uint8_t *tile, int rows, int r, int c, float x, float y) {
    *reinterpret_cast<uint32_t *>(tile + sw_off(rows, r, c)) = tc::pack_bf16x2(x, y);
}

// A fragment of rows [m0, m0+16) x columns [k0, k0+16) of A^T, read from a tile stored [k][m]
// (the transposed operand), through the transposing load.
__device__ __forceinline__ void load_a_t(uint32_t base, int rows, int m0, int k0, uint32_t (&a)[4]) {
    const int lane = threadIdx.x & 31;
    ldsm4t(base + sw_off(rows, k0 + (lane & 7) + ((lane >> 4) << 3), m0 + (((lane >> 3) & 1) << 3)), a);
}

}  // namespace wmma16
}  // namespace bla
