// Weight repacking at init: row-major [M, K] -> the tile-packed layout the streaming
// kernels read (fe_stream.cuh). Tile (g, s) holds rows 4g..4g+3 and columns
// [s*KS, s*KS + w), w = min(KS, K - s*KS), stored row after row (row stride w), so one
// pipeline stage is one contiguous bulk copy. Rows past M (the last group's padding) are
// zero. Works in 16-byte vectors; K * element size must be a multiple of 16.
#include "fe_kernels.h"
#include "fe_stream.cuh"

namespace fe {

__global__ void pack_tiles_kernel(const uint4* __restrict__ src, uint4* __restrict__ dst, int M, int Kv, int KSv,
                                  int64_t total) {
    for (int64_t q = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; q < total;
         q += (int64_t)gridDim.x * blockDim.x) {
        const int64_t per_group = (int64_t)kGroupRows * Kv;
        const int g = (int)(q / per_group);
        const int rem = (int)(q - (int64_t)g * per_group);
        const int s = rem / (kGroupRows * KSv);
        const int rem2 = rem - s * kGroupRows * KSv;
        const int w = min(KSv, Kv - s * KSv);
        const int r = rem2 / w, c = rem2 - r * w;
        const int row = g * kGroupRows + r;
        dst[q] = row < M ? src[(int64_t)row * Kv + (int64_t)s * KSv + c] : make_uint4(0, 0, 0, 0);
    }
}

size_t packed_bytes(int M, int K, int es) {
    return (size_t)((M + kGroupRows - 1) / kGroupRows) * kGroupRows * K * es;
}

cudaError_t launch_pack_tiles(const void* src, void* dst, int M, int K, int es, cudaStream_t st) {
    const int Kv = K * es / 16;
    const int KSv = kTileBytes / (kGroupRows * 16);  // 16-byte vectors per row of a full slice
    const int64_t total = (int64_t)packed_bytes(M, K, es) / 16;
    const int blocks = (int)((total + 255) / 256 < 4096 ? (total + 255) / 256 : 4096);
    pack_tiles_kernel<<<blocks, 256, 0, st>>>((const uint4*)src, (uint4*)dst, M, Kv, KSv, total);
    return cudaGetLastError();
}

}  // namespace fe

// ---- tensor-core layout -------------------------------------------------------------------
// [ceil(M/128)][K/64] blocks of 128 rows x 64 bf16, each block 16 KB in the 128B-swizzled
// K-major layout of fe_tc.cuh (row r, 16-byte chunk c at sw128_offset(r, c)); rows past M
// are zero. One block is the A operand of four M=128, K=16 MMAs.
namespace fe {

__global__ void pack_mma_kernel(const uint4* __restrict__ src, uint4* __restrict__ dst, int M, int K, int64_t total) {
    const int nkb = K / 64;
    for (int64_t q = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; q < total;
         q += (int64_t)gridDim.x * blockDim.x) {
        const int64_t blk = q / 1024;  // 1024 chunks of 16 B per block
        const int within = (int)(q - blk * 1024);
        const int tile = (int)(blk / nkb), kb = (int)(blk - (int64_t)tile * nkb);
        const int atom = within / 64, rin = (within / 8) % 8, pch = within % 8;
        const int row = atom * 8 + rin, chunk = pch ^ rin;
        const int64_t m = (int64_t)tile * 128 + row;
        dst[q] = m < M ? src[m * (K / 8) + (int64_t)kb * 8 + chunk] : make_uint4(0, 0, 0, 0);
    }
}

size_t mma_packed_bytes(int M, int K) { return (size_t)((M + 127) / 128) * 128 * K * 2; }

cudaError_t launch_pack_mma(const void* src, void* dst, int M, int K, cudaStream_t st) {
    const int64_t total = (int64_t)mma_packed_bytes(M, K) / 16;
    const int blocks = (int)((total + 255) / 256 < 4096 ? (total + 255) / 256 : 4096);
    pack_mma_kernel<<<blocks, 256, 0, st>>>((const uint4*)src, (uint4*)dst, M, K, total);
    return cudaGetLastError();
}

}  // namespace fe
