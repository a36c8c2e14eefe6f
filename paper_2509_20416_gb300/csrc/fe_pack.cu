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
