// synth_gpu.cu -- GPU twin of synth/__init__.py (seeded synthetic inputs).
//
// Input generation only: no part of the method runs here.  Produces bf16 rows
// bit-identical to the numpy generator (integer SplitMix64 words, Irwin-Hall
// sum of twelve 16-bit uniforms, one optional fp32 scale multiply, RNE to
// bf16), so that full-size caches can be filled on the device while the CPU
// side regenerates any sampled row from its position alone.
#include <cuda_runtime.h>
#include <stdint.h>

namespace {

__device__ __forceinline__ uint64_t sm64_mix(uint64_t z)
{
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

__device__ __forceinline__ uint16_t synth_value(uint64_t seed, uint64_t stream, uint64_t layer, uint64_t seq,
                                                uint64_t head, uint64_t pos, uint64_t ch, const float* scale)
{
    uint64_t i = ((((((stream << 8) | layer) << 12 | seq) << 8 | head) << 20 | pos) << 7) | ch;
    int64_t total = 0;
    for (int k = 0; k < 3; ++k) {
        uint64_t w = sm64_mix(seed + (3ull * i + (uint64_t)(k + 1)) * 0x9E3779B97F4A7C15ull);
        total += (int64_t)(w & 0xFFFF) + (int64_t)((w >> 16) & 0xFFFF) + (int64_t)((w >> 32) & 0xFFFF) +
                 (int64_t)((w >> 48) & 0xFFFF);
    }
    int32_t n = (int32_t)(total - 6 * 65535);
    float f = __fmul_rn((float)n, 1.0f / 65536.0f);
    if (scale) f = __fmul_rn(f, *scale);
    uint32_t b = __float_as_uint(f);
    b = b + 0x7FFFu + ((b >> 16) & 1u);
    return (uint16_t)(b >> 16);
}

// out[b][h][i][ch] = value(seed, stream, layer, seq0 + b, h, pos[b][h][i], ch); pos < 0 -> zero row.
__global__ void synth_rows_kernel(uint16_t* __restrict__ out, const int32_t* __restrict__ pos, int B, int NH,
                                  int n, int d, uint64_t seed, int stream, int layer, int seq0,
                                  const float* __restrict__ scale /* [NH][d] or null */)
{
    const long long total = (long long)B * NH * n * d;
    for (long long e = (long long)blockIdx.x * blockDim.x + threadIdx.x; e < total;
         e += (long long)gridDim.x * blockDim.x) {
        const int ch = (int)(e % d);
        const long long row = e / d;
        const int h = (int)((row / n) % NH);
        const int b = (int)(row / ((long long)n * NH));
        const int p = pos[row];
        uint16_t v = 0;
        if (p >= 0)
            v = synth_value(seed, (uint64_t)stream, (uint64_t)layer, (uint64_t)(seq0 + b), (uint64_t)h,
                            (uint64_t)p, (uint64_t)ch, scale ? scale + (size_t)h * d + ch : nullptr);
        out[e] = v;
    }
}

} // namespace

extern "C" {

// Fills out[B][NH][n][d] (bf16 bits) from positions pos[B][NH][n] (device
// pointers).  Returns 0, or a CUDA error code.  Asynchronous on `stream`.
int synth_fill_rows(void* out, const int32_t* pos, int B, int NH, int n, int d, uint64_t seed, int stream_id,
                    int layer, int seq0, const float* scale, void* stream)
{
    if (!out || !pos || B <= 0 || NH <= 0 || n <= 0 || d <= 0 || d > 128) return 1;
    long long total = (long long)B * NH * n * d;
    long long blocks = (total + 255) / 256;
    if (blocks > 152LL * 64) blocks = 152LL * 64;
    synth_rows_kernel<<<(unsigned)blocks, 256, 0, (cudaStream_t)stream>>>(
        (uint16_t*)out, pos, B, NH, n, d, seed, stream_id, layer, seq0, scale);
    return (int)cudaGetLastError();
}

} // extern "C"
