// rheo_device.cuh -- device building blocks of the RheoSampling kernels (sm_103a).
//
// Row streaming: a row of V logits is cut into chunks of kChunkBytes; one CTA
// of kThreads threads loads a chunk with kNV 128-bit loads per thread (element
// e of the chunk lives in thread (e / VEC) % kThreads, load (e / VEC) / kThreads),
// so a warp's load instruction covers 512 contiguous bytes.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace rheo {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kNV = 8;                                 // 128-bit loads per thread per chunk
constexpr int kChunkBytes = kThreads * kNV * 16;       // 32 KiB per CTA
constexpr int kMaxSupport = 128;
constexpr int kCandCap = 2048;                         // per-chunk candidate buffer (keys)
constexpr int kMaxVocab = 262144;
constexpr int kMaxNodes = 16384;

enum : uint32_t {
    kStBadLogit = 1u,
    kStEmptyRow = 2u,
    kStBadTemperature = 4u,
    kStInternal = 8u,
};

enum : int { kTagSample = 1, kTagVerify = 2, kTagResidual = 3 };
enum : uint8_t { kSlotRoot = 0, kSlotLead = 1, kSlotSampled = 2, kSlotFill = 3 };

// ---------------------------------------------------------------------------
// element types: DT 0 = fp32 (4 per 16 B), DT 1 = bf16 (8 per 16 B)
// ---------------------------------------------------------------------------
template <int DT> struct Elem;
template <> struct Elem<0> {
    static constexpr int VEC = 4;
    static constexpr int SIZE = 4;
    static constexpr int CHUNK = kChunkBytes / 4;
    // raw 32-bit pattern of element i of a 16-byte vector
    __device__ static __forceinline__ uint32_t raw(const uint4& v, int i) {
        return i == 0 ? v.x : i == 1 ? v.y : i == 2 ? v.z : v.w;
    }
    __device__ static __forceinline__ float value(uint32_t r) { return __uint_as_float(r); }
    // order-preserving 32-bit key; -0 and +0 share a key
    __device__ static __forceinline__ uint32_t key(uint32_t r) {
        if (r == 0x80000000u) r = 0u;
        return (r & 0x80000000u) ? ~r : (r | 0x80000000u);
    }
    __device__ static __forceinline__ float value_of_key(uint32_t k) {
        uint32_t r = (k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k;
        return __uint_as_float(r);
    }
    __device__ static __forceinline__ uint32_t neg_inf_raw() { return 0xFF800000u; }
    __device__ static __forceinline__ uint32_t load_scalar(const char* row, int64_t e) {
        return __ldg(reinterpret_cast<const uint32_t*>(row) + e);
    }
};
template <> struct Elem<1> {
    static constexpr int VEC = 8;
    static constexpr int SIZE = 2;
    static constexpr int CHUNK = kChunkBytes / 2;
    __device__ static __forceinline__ uint32_t raw(const uint4& v, int i) {
        uint32_t w = (i >> 1) == 0 ? v.x : (i >> 1) == 1 ? v.y : (i >> 1) == 2 ? v.z : v.w;
        return (i & 1) ? (w >> 16) : (w & 0xFFFFu);
    }
    __device__ static __forceinline__ float value(uint32_t r) { return __uint_as_float(r << 16); }
    // bf16 keys keep the 16 significant bits on top (low half zero)
    __device__ static __forceinline__ uint32_t key(uint32_t r) {
        if (r == 0x8000u) r = 0u;
        uint32_t k = (r & 0x8000u) ? (~r & 0xFFFFu) : (r | 0x8000u);
        return k << 16;
    }
    __device__ static __forceinline__ float value_of_key(uint32_t k) {
        uint32_t h = k >> 16;
        h = (h & 0x8000u) ? (h & 0x7FFFu) : (~h & 0xFFFFu);
        return __uint_as_float(h << 16);
    }
    __device__ static __forceinline__ uint32_t neg_inf_raw() { return 0xFF80u; }
    __device__ static __forceinline__ uint32_t load_scalar(const char* row, int64_t e) {
        return (uint32_t)__ldg(reinterpret_cast<const unsigned short*>(row) + e);
    }
};

__device__ __forceinline__ uint4 ld_stream(const void* p) {
    uint4 r;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(p));
    return r;
}

// 16 bytes holding elements [e0, e0 + VEC) of a row; elements >= V read as -inf.
template <int DT, bool ALIGNED>
__device__ __forceinline__ uint4 load_vec(const char* row, int64_t e0, int V) {
    using E = Elem<DT>;
    if (ALIGNED && e0 + E::VEC <= V) return ld_stream(row + e0 * E::SIZE);
    uint32_t w[E::VEC];
#pragma unroll
    for (int i = 0; i < E::VEC; ++i) w[i] = (e0 + i < V) ? E::load_scalar(row, e0 + i) : E::neg_inf_raw();
    uint4 r;
    if (DT == 0) {
        r.x = w[0]; r.y = w[1]; r.z = w[2]; r.w = w[3];
    } else {
        r.x = w[0] | (w[1] << 16);
        r.y = w[2] | (w[3] << 16);
        r.z = w[4 % E::VEC] | (w[5 % E::VEC] << 16);
        r.w = w[6 % E::VEC] | (w[7 % E::VEC] << 16);
    }
    return r;
}

// 2^x on the special-function unit (used only inside partition sums)
__device__ __forceinline__ float fast_exp2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ uint32_t ord_f32(float x) { return Elem<0>::key(__float_as_uint(x)); }

// ---------------------------------------------------------------------------
// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11) and the uniform map
// key = (lo32 seed, hi32 seed); counter = (draw>>2, lo32 offset, 4*node+tag, hi32 offset)
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        const uint32_t lo0 = 0xD2511F53u * c.x, hi0 = __umulhi(0xD2511F53u, c.x);
        const uint32_t lo1 = 0xCD9E8D57u * c.z, hi1 = __umulhi(0xCD9E8D57u, c.z);
        c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
        k0 += 0x9E3779B9u;
        k1 += 0xBB67AE85u;
    }
    return c;
}

__device__ __forceinline__ uint4 philox_block(uint64_t seed, uint64_t offset, int tag, int node, uint64_t draw4) {
    return philox4x32_10(make_uint4((uint32_t)draw4, (uint32_t)offset, (uint32_t)(4 * node + tag),
                                    (uint32_t)(offset >> 32)),
                         (uint32_t)seed, (uint32_t)(seed >> 32));
}

__device__ __forceinline__ uint32_t word_of(const uint4& r, int i) {
    return i == 0 ? r.x : i == 1 ? r.y : i == 2 ? r.z : r.w;
}

// ((w >> 9) + 0.5) * 2^-23: exact in fp32, strictly inside (0, 1)
__device__ __forceinline__ float u01(uint32_t w) {
    return __fmul_rn(__fadd_rn((float)(w >> 9), 0.5f), 1.0f / 8388608.0f);
}

__device__ __forceinline__ float uniform(uint64_t seed, uint64_t offset, int tag, int node, uint64_t draw) {
    return u01(word_of(philox_block(seed, offset, tag, node, draw >> 2), (int)(draw & 3)));
}

__device__ __forceinline__ float gumbel(float u) { return -logf(-logf(u)); }

// ---------------------------------------------------------------------------
// block reductions (kThreads threads, all must call)
// ---------------------------------------------------------------------------
struct BlockScratch {
    int ired[2][kWarps];
    double dred[kWarps];
    float fred[kWarps];
    unsigned long long ured[kWarps];
    int flag;
};

__device__ __forceinline__ int block_sum_int(int v, BlockScratch& s, int& parity) {
    v = __reduce_add_sync(0xFFFFFFFFu, v);
    int* buf = s.ired[parity];
    parity ^= 1;
    if ((threadIdx.x & 31) == 0) buf[threadIdx.x >> 5] = v;
    __syncthreads();
    int t = 0;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) t += buf[w];
    return t;
}

__device__ __forceinline__ unsigned long long warp_max_u64(unsigned long long v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        unsigned long long w = __shfl_xor_sync(0xFFFFFFFFu, v, o);
        v = w > v ? w : v;
    }
    return v;
}

__device__ __forceinline__ unsigned long long block_max_u64(unsigned long long v, BlockScratch& s) {
    v = warp_max_u64(v);
    __syncthreads();
    if ((threadIdx.x & 31) == 0) s.ured[threadIdx.x >> 5] = v;
    __syncthreads();
    unsigned long long t = 0;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) t = s.ured[w] > t ? s.ured[w] : t;
    return t;
}

__device__ __forceinline__ unsigned long long block_and_or_u64(unsigned long long v, bool want_or,
                                                               BlockScratch& s) {
    unsigned lo = (unsigned)v, hi = (unsigned)(v >> 32);
    if (want_or) {
        lo = __reduce_or_sync(0xFFFFFFFFu, lo);
        hi = __reduce_or_sync(0xFFFFFFFFu, hi);
    } else {
        lo = __reduce_and_sync(0xFFFFFFFFu, lo);
        hi = __reduce_and_sync(0xFFFFFFFFu, hi);
    }
    v = ((unsigned long long)hi << 32) | lo;
    __syncthreads();
    if ((threadIdx.x & 31) == 0) s.ured[threadIdx.x >> 5] = v;
    __syncthreads();
    unsigned long long t = want_or ? 0ull : ~0ull;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) t = want_or ? (t | s.ured[w]) : (t & s.ured[w]);
    return t;
}

// (max, sum of exp relative to max): merged in fp64
__device__ __forceinline__ void block_max_sum(float mu, double sum, BlockScratch& s, float& out_mu,
                                              double& out_sum) {
    float m = mu;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
    __syncthreads();
    if ((threadIdx.x & 31) == 0) s.fred[threadIdx.x >> 5] = m;
    __syncthreads();
    float M = s.fred[0];
#pragma unroll
    for (int w = 1; w < kWarps; ++w) M = fmaxf(M, s.fred[w]);
    double t = (sum > 0.0) ? sum * exp((double)mu - (double)M) : 0.0;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xFFFFFFFFu, t, o);
    if ((threadIdx.x & 31) == 0) s.dred[threadIdx.x >> 5] = t;
    __syncthreads();
    double T = 0.0;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) T += s.dred[w];
    out_mu = M;
    out_sum = T;
}

// ---------------------------------------------------------------------------
// Selection: the k-th largest of a set of 64-bit keys spread over the block.
// count_ge(t) returns how many of the calling thread's keys are >= t.  and_all
// / or_all are the bitwise AND / OR of every key.  Returns a threshold T with
// count(keys >= T) == k when keys are distinct (and the k-th largest value when
// they are not).  Bits that are equal in every key are copied without a step.
// ---------------------------------------------------------------------------
template <class CountGE>
__device__ unsigned long long block_select(CountGE count_ge, int k, unsigned long long and_all,
                                           unsigned long long or_all, BlockScratch& s, int& parity) {
    unsigned long long prefix = 0;
    const unsigned long long fixed = ~(and_all ^ or_all);
    for (int bit = 63; bit >= 0; --bit) {
        const unsigned long long mask = 1ull << bit;
        if (fixed & mask) {
            prefix |= (and_all & mask);
            continue;
        }
        const unsigned long long t = prefix | mask;
        const int c = block_sum_int(count_ge(t), s, parity);
        if (c >= k) {
            prefix = t;
            if (c == k) return prefix;
        }
    }
    return prefix;
}

// exclusive prefix sum over the block (in thread order)
__device__ __forceinline__ int block_exclusive_scan(int v, int& total, BlockScratch& s) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        int y = __shfl_up_sync(0xFFFFFFFFu, x, o);
        if (lane >= o) x += y;
    }
    __syncthreads();
    if (lane == 31) s.ired[0][warp] = x;
    __syncthreads();
    int before = 0;
    total = 0;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) {
        if (w < warp) before += s.ired[0][w];
        total += s.ired[0][w];
    }
    __syncthreads();
    return before + x - v;
}

// Arrival counter for "last CTA of a group" hand-off.  Never waits: the CTA
// that arrives last does the follow-up work and resets the counter.
__device__ __forceinline__ bool arrive_last(unsigned* counter, unsigned total, BlockScratch& s) {
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) {
        const unsigned prev = atomicAdd(counter, 1u);
        s.flag = (prev == total - 1) ? 1 : 0;
        if (s.flag) *counter = 0u;
    }
    __syncthreads();
    const bool last = s.flag != 0;
    if (last) __threadfence();
    return last;
}

// numbering helpers (see rheo.h)
__device__ __forceinline__ int64_t depth_base(int K, int d) {
    return d == 1 ? 1 : 1 + (int64_t)(K + 1) + (int64_t)(d - 2) * K * (K + 1);
}
__device__ __forceinline__ int slot_of(int K, int64_t g) {
    if (g <= K + 1) return (int)(g - 1);
    return (int)((g - (K + 2)) % (K + 1));
}
__device__ __forceinline__ int64_t parent_expansion_of(int K, int64_t g) {
    if (g <= K + 1) return 0;
    const int64_t w = g - (K + 2), per = (int64_t)K * (K + 1);
    return 1 + (w / per) * K + (w % per) / (K + 1);
}
__device__ __forceinline__ int depth_of(int K, int64_t g) {
    if (g == 0) return 0;
    if (g <= K + 1) return 1;
    return 2 + (int)((g - (K + 2)) / ((int64_t)K * (K + 1)));
}

}  // namespace rheo
