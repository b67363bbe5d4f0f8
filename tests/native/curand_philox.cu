// Test helper: Philox4x32-10 blocks from cuRAND's device generator, used as
// an independent check of libpps's keyed source.  cuRAND's state holds a
// 128-bit counter (offset/4 in words 0-1, subsequence in words 2-3) and a
// 64-bit key (the seed); curand4 returns the four words of the current block.
#include <cstdint>
#include <curand_kernel.h>

__global__ void curand_blocks_kernel(const uint32_t* ctr, const uint32_t* key, uint32_t* out, int n) {
    int t = blockIdx.x * blockDim.x + threadIdx.x;
    if (t >= n) return;
    unsigned long long seed = (unsigned long long)key[2 * t] | ((unsigned long long)key[2 * t + 1] << 32);
    unsigned long long subseq = (unsigned long long)ctr[4 * t + 2] | ((unsigned long long)ctr[4 * t + 3] << 32);
    unsigned long long blk = (unsigned long long)ctr[4 * t] | ((unsigned long long)ctr[4 * t + 1] << 32);
    curandStatePhilox4_32_10_t st;
    curand_init(seed, subseq, 4ull * blk, &st);
    uint4 r = curand4(&st);
    out[4 * t] = r.x;
    out[4 * t + 1] = r.y;
    out[4 * t + 2] = r.z;
    out[4 * t + 3] = r.w;
}

extern "C" int curand_philox_blocks(const uint32_t* ctr, const uint32_t* key, uint32_t* out, int n, void* stream) {
    if (n <= 0) return 0;
    curand_blocks_kernel<<<(n + 127) / 128, 128, 0, (cudaStream_t)stream>>>(ctr, key, out, n);
    return (int)cudaGetLastError();
}
