/*
 * Host (CPU) implementation of the seeded input generator of mlkv_synth/gen.py, for the large row
 * samples of the full-size parity tests.  Same definition as gen.py and synth_gpu.cu; holds no
 * attention arithmetic.
 *
 *   void synth_host_fill_bf16(uint16_t* dst, long long rows, long long cols, long long pitch,
 *                             const long long* row_ids, long long col0, unsigned long long seed,
 *                             unsigned long long tensor_id, float sigma)
 *   dst[r*pitch + c] = bf16 bits of value(row_ids[r], col0 + c)
 */
#include <stdint.h>
#include <string.h>

static const uint64_t kGamma = 0x9E3779B97F4A7C15ull;

static uint64_t mix64(uint64_t z)
{
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

static uint64_t sm_out(uint64_t s, uint64_t n) { return mix64(s + (n + 1) * kGamma); }

static uint32_t sum16(uint64_t x)
{
    return (uint32_t)((x & 0xffff) + ((x >> 16) & 0xffff) + ((x >> 32) & 0xffff) + (x >> 48));
}

static uint16_t f32_to_bf16_rne(float f)
{
    uint32_t b;
    memcpy(&b, &f, 4);
    b = b + 0x7fffu + ((b >> 16) & 1u);
    return (uint16_t)(b >> 16);
}

void synth_host_fill_bf16(uint16_t *dst, long long rows, long long cols, long long pitch,
                          const long long *row_ids, long long col0, unsigned long long seed,
                          unsigned long long tensor_id, float sigma)
{
    const uint64_t s_tensor = sm_out(seed, tensor_id);
    for (long long r = 0; r < rows; ++r) {
        const uint64_t s_row = sm_out(s_tensor, (uint64_t)row_ids[r]);
        uint16_t *out = dst + r * pitch;
        for (long long c = 0; c < cols; ++c) {
            const uint64_t n = 3ull * (uint64_t)(col0 + c);
            const uint32_t total = sum16(sm_out(s_row, n)) + sum16(sm_out(s_row, n + 1)) +
                                   sum16(sm_out(s_row, n + 2));
            const float z = (float)((int)total - 6 * 65536) * (1.0f / 65536.0f);
            out[c] = f32_to_bf16_rne(sigma * z);
        }
    }
}
