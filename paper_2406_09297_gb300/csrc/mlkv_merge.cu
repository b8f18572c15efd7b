// KV-weight merging by averaging (Sec. 4.2) on GB300: MHA K or V projection weights become MLKV's
// (m owner layers) x (g KV heads).  Merged head j of owner layer o is the mean, over every layer n
// of o's block (owner[n] == o) and every head i of group j (Eq. 12), of that head's rows; the
// result is rounded to bf16, to nearest with ties to even.
//
// HBM-bound: every input element is read once, every output element written once.  A thread owns
// 8 consecutive elements (16 bytes) of one merged head and walks its members (or a slice of them,
// when the weights are too small to fill the GPU otherwise; the slices' sums are then folded).
//
// The mean without FP64 (GB300 adds doubles at a few per clock per SM, less than HBM delivers):
// each column's sum is kept as an unevaluated pair of floats, hi + lo, where TwoSum (Knuth)
// returns every addition's rounding error exactly and lo collects the errors; the pair is divided
// by the member count with an FMA-exact remainder, renormalised, and rounded to bf16 with lo
// deciding the ties of hi.  The result is the bf16 nearest to the exact mean unless that mean lies
// within about n^2 2^-48 (relative) of a bf16 rounding boundary, n the member count.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "mlkv_internal.h"

namespace mlkv {
namespace {

// s + e == a + b exactly, for two columns at once (round-to-nearest; x - y is fma(y, -1, x),
// which rounds once, like the subtraction).
__device__ __forceinline__ void two_sum2(float2 a, float2 b, float2 &s, float2 &e)
{
    const float2 m1 = make_float2(-1.f, -1.f);
    s = __fadd2_rn(a, b);
    const float2 bv = __ffma2_rn(a, m1, s);    // s - a
    const float2 av = __ffma2_rn(bv, m1, s);   // s - bv
    e = __fadd2_rn(__ffma2_rn(av, m1, a), __ffma2_rn(bv, m1, b));
}

__device__ __forceinline__ void acc_add2(float2 &hi, float2 &lo, float2 x)
{
    float2 s, e;
    two_sum2(hi, x, s, e);
    hi = s;
    lo = __fadd2_rn(lo, e);
}

// The two bf16 of a word, low half first, as floats (exact).
__device__ __forceinline__ float2 unpack_bf16x2(uint32_t w)
{
    return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xFFFF0000u));
}

__device__ __forceinline__ void two_sum(float a, float b, float &s, float &e)
{
    s = __fadd_rn(a, b);
    const float bv = __fsub_rn(s, a);
    const float av = __fsub_rn(s, bv);
    e = __fadd_rn(__fsub_rn(a, av), __fsub_rn(b, bv));
}

// bf16 bits nearest to the pair's value hi + lo (|lo| at most half a float ulp of hi).
__device__ __forceinline__ uint32_t round_pair_bf16(float hi, float lo)
{
    const uint32_t b = __float_as_uint(hi);
    if ((b & 0x7F800000u) == 0x7F800000u)   // inf or NaN
        return (b & 0x007FFFFFu) ? 0x7FC0u : (b >> 16);
    const uint32_t low = b & 0xFFFFu;
    uint32_t up;
    if (low != 0x8000u)
        up = low > 0x8000u;
    else if (lo != 0.f)
        up = (lo > 0.f) == (hi > 0.f);   // past the tie in magnitude
    else
        up = (b >> 16) & 1u;              // an exact tie: to even
    return ((b & 0xFFFF0000u) + (up << 16)) >> 16;
}

// (hi + lo) / count rounded to bf16: q1 the rounded quotient of hi, hi - q1 count exact (FMA).
__device__ __forceinline__ uint32_t mean_bf16(float hi, float lo, float count)
{
    const float q1 = __fdiv_rn(hi, count);
    const float r = __fadd_rn(__fmaf_rn(-q1, count, hi), lo);
    const float q2 = __fdiv_rn(r, count);
    float qh, ql;
    two_sum(q1, q2, qh, ql);
    return round_pair_bf16(qh, ql);
}

// S slices of a CTA split one head's members; each thread owns 8 columns (16 bytes).
template <int S>
__global__ void __launch_bounds__(256) merge_kernel(const __grid_constant__ MergeParams p)
{
    constexpr int kVec = 256 / S;                // 16-byte column groups per CTA pass
    __shared__ float2 part[S > 1 ? S - 1 : 1][kVec][8];   // slices 1.. : hi pairs, lo pairs
    const int slice = threadIdx.x / kVec;
    const int tv = threadIdx.x - slice * kVec;
    // One CTA per (merged head, chunk of kVec column groups), chunks of a head consecutive: the
    // CTAs resident at a time stream a few megabytes of a few heads' rows, not scattered pages.
    const long long chunks = ((p.row >> 3) + kVec - 1) / kVec;
    const int sj = static_cast<int>(blockIdx.x / chunks);   // slot * g + j
    const long long base = (static_cast<long long>(blockIdx.x) - sj * chunks) * kVec;
    const int s = sj / p.g;
    const int j = sj - s * p.g;
    const long long nvec = p.row >> 3;
    const int b0 = p.slot_begin[s];
    const int members = (p.slot_begin[s + 1] - b0) * p.G;   // (layer, head) pairs
    const int m0 = static_cast<int>(static_cast<long long>(members) * slice / S);
    const int m1 = static_cast<int>(static_cast<long long>(members) * (slice + 1) / S);
    const float count = static_cast<float>(members);
    const size_t head_stride = static_cast<size_t>(p.row);
    {
        const long long v = base + tv;
        float2 hi[4], lo[4];
#pragma unroll
        for (int c = 0; c < 4; ++c)
            hi[c] = lo[c] = make_float2(0.f, 0.f);
        if (v < nvec && m0 < m1) {
            // Members in order: heads j*G .. j*G+G-1 of each layer of the block.  Walk them with a
            // pointer and a head counter (no division per load).
            const size_t col = static_cast<size_t>(v) * 8;
            int lk = m0 / p.G;                   // member layer index
            int hk = m0 - lk * p.G;              // head within the group
            auto layer_ptr = [&](int k) {
                return p.W + (static_cast<size_t>(p.member[b0 + k]) * p.h +
                              static_cast<size_t>(j) * p.G) * head_stride + col;
            };
            const __nv_bfloat16 *ptr = layer_ptr(lk) + hk * head_stride;
            auto next = [&]() {
                const __nv_bfloat16 *cur = ptr;
                if (++hk == p.G) {
                    hk = 0;
                    ++lk;
                    if (b0 + lk < p.slot_begin[s + 1])
                        ptr = layer_ptr(lk);
                } else {
                    ptr += head_stride;
                }
                return reinterpret_cast<const uint4 *>(cur);
            };
            int mi = m0;
            for (; mi + 4 <= m1; mi += 4) {
                uint4 w[4];
#pragma unroll
                for (int u = 0; u < 4; ++u)   // four loads in flight before any addition
                    w[u] = __ldcs(next());
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    acc_add2(hi[0], lo[0], unpack_bf16x2(w[u].x));
                    acc_add2(hi[1], lo[1], unpack_bf16x2(w[u].y));
                    acc_add2(hi[2], lo[2], unpack_bf16x2(w[u].z));
                    acc_add2(hi[3], lo[3], unpack_bf16x2(w[u].w));
                }
            }
            for (; mi < m1; ++mi) {
                const uint4 w = __ldcs(next());
                acc_add2(hi[0], lo[0], unpack_bf16x2(w.x));
                acc_add2(hi[1], lo[1], unpack_bf16x2(w.y));
                acc_add2(hi[2], lo[2], unpack_bf16x2(w.z));
                acc_add2(hi[3], lo[3], unpack_bf16x2(w.w));
            }
        }
        if (S > 1) {
            // Slices 1.. hand their pairs to slice 0, which folds them in slice order.
            if (slice > 0) {
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    part[slice - 1][tv][c] = hi[c];
                    part[slice - 1][tv][4 + c] = lo[c];
                }
            }
            __syncthreads();
            if (slice == 0) {
#pragma unroll
                for (int k = 0; k < S - 1; ++k)
#pragma unroll
                    for (int c = 0; c < 4; ++c) {
                        float2 sum, e;
                        two_sum2(hi[c], part[k][tv][c], sum, e);
                        hi[c] = sum;
                        lo[c] = __fadd2_rn(__fadd2_rn(lo[c], e), part[k][tv][4 + c]);
                    }
            }
            __syncthreads();
        }
        if (slice == 0 && v < nvec) {
            uint4 out;
            out.x = mean_bf16(hi[0].x, lo[0].x, count) | (mean_bf16(hi[0].y, lo[0].y, count) << 16);
            out.y = mean_bf16(hi[1].x, lo[1].x, count) | (mean_bf16(hi[1].y, lo[1].y, count) << 16);
            out.z = mean_bf16(hi[2].x, lo[2].x, count) | (mean_bf16(hi[2].y, lo[2].y, count) << 16);
            out.w = mean_bf16(hi[3].x, lo[3].x, count) | (mean_bf16(hi[3].y, lo[3].y, count) << 16);
            __stcs(reinterpret_cast<uint4 *>(p.out + static_cast<size_t>(sj) * head_stride +
                                             static_cast<size_t>(v) * 8),
                   out);
        }
    }
}

}  // namespace

cudaError_t launch_merge(const MergeParams &p, int n_slots, cudaStream_t stream)
{
    // Split each head's members over S slices while the (head, column group) work alone would
    // leave the SMs short of the ~2 k threads each keeps resident.
    const long long nvec = p.row >> 3;
    const int sj = n_slots * p.g;
    const long long target = 152LL * 2048;
    int max_members = 0;
    for (int s = 0; s < n_slots; ++s)
        max_members = max(max_members, (p.slot_begin[s + 1] - p.slot_begin[s]) * p.G);
    int S = 1;
    while (S < 8 && nvec * sj * S < target && max_members >= 4 * 2 * S)
        S *= 2;
    const long long chunks = (nvec + 256 / S - 1) / (256 / S);
    if (chunks * sj > 0x7FFFFFFFLL)
        return cudaErrorInvalidConfiguration;
    const dim3 grid(static_cast<unsigned>(chunks * sj));
    switch (S) {
    case 1: merge_kernel<1><<<grid, 256, 0, stream>>>(p); break;
    case 2: merge_kernel<2><<<grid, 256, 0, stream>>>(p); break;
    case 4: merge_kernel<4><<<grid, 256, 0, stream>>>(p); break;
    default: merge_kernel<8><<<grid, 256, 0, stream>>>(p); break;
    }
    return cudaGetLastError();
}

}  // namespace mlkv
