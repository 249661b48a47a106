// rheo_device.cuh -- device building blocks of the RheoSampling kernels (sm_103a).
//
// Row streaming: a row of V logits is cut into chunks of kChunkBytes; one CTA
// of kThreads threads loads a chunk with kNV 128-bit loads per thread (element
// e of the chunk lives in thread (e / VEC) % kThreads, load (e / VEC) / kThreads),
// so a warp's load instruction covers 512 contiguous bytes.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace rheo {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kMaxWarps = 16;  // largest block of the path (512 threads); scratch is sized for it
constexpr int kNV = 8;                                 // 128-bit loads per thread per chunk
constexpr int kChunkBytes = kThreads * kNV * 16;       // 32 KiB per CTA
constexpr int kMaxSupport = 128;
constexpr int kCandCap = 2048;                         // per-chunk candidate buffer (keys)
constexpr int kMaxVocab = 262144;
constexpr int kMaxNodes = 16384;

// Programmatic dependent launch: every kernel of the path first waits until
// the grid before it on the stream has completed and its writes are visible
// (a no-op when launched without the programmatic attribute), then lets the
// next grid start launching, so launch latency overlaps the end of this one.
__device__ __forceinline__ void grid_dependency_begin() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

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
    // key of a value read from this element type
    __device__ static __forceinline__ uint32_t key_of_value(float x) { return key(__float_as_uint(x)); }
    // value with the same order as a threshold key; keys at or below key(-inf) give -inf
    __device__ static __forceinline__ float threshold_value(uint32_t k) {
        return k <= 0x007FFFFFu ? -INFINITY : value_of_key(k);
    }
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
    __device__ static __forceinline__ uint32_t key_of_value(float x) { return key(__float_as_uint(x) >> 16); }
    __device__ static __forceinline__ float threshold_value(uint32_t k) {
        return k <= 0x007F0000u ? -INFINITY : value_of_key(k);
    }
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

// Pairs of fp32 values in one 64-bit register, operated on two at a time by the
// packed fp32 instructions of sm_100+ (same per-element rounding as the scalar
// fma / add / mul).
__device__ __forceinline__ unsigned long long f2_pack(float a, float b) {
    unsigned long long r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a), "f"(b));
    return r;
}
__device__ __forceinline__ float f2_fold(unsigned long long x) {  // a + b
    float a, b;
    asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(x));
    return a + b;
}
__device__ __forceinline__ unsigned long long f2_fma(unsigned long long a, unsigned long long b, unsigned long long c) {
    unsigned long long r;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
    return r;
}
__device__ __forceinline__ unsigned long long f2_add(unsigned long long a, unsigned long long b) {
    unsigned long long r;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}
__device__ __forceinline__ unsigned long long f2_mul(unsigned long long a, unsigned long long b) {
    unsigned long long r;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}
// (2^a, 2^b) of a pair
__device__ __forceinline__ unsigned long long f2_exp2(unsigned long long x) {
    float a, b;
    asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(x));
    return f2_pack(fast_exp2(a), fast_exp2(b));
}

// ---------------------------------------------------------------------------
// 16-byte vectors of logits: max, partition-sum terms, tail masking
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t bmax2(uint32_t a, uint32_t b) {
    uint32_t r;
    asm("max.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
    return r;
}
__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

template <int DT> struct Vec;
template <> struct Vec<1> {
    __device__ static __forceinline__ float vmax(const uint4& v) {
        const uint32_t m = bmax2(bmax2(v.x, v.y), bmax2(v.z, v.w));
        return fmaxf(bf_lo(m), bf_hi(m));
    }
    // sum of 2^(x c - mc) over the 8 values (independent partial sums)
    __device__ static __forceinline__ float vexp(const uint4& v, float c, float mc) {
        const float a0 = fast_exp2(fmaf(bf_lo(v.x), c, -mc)) + fast_exp2(fmaf(bf_hi(v.x), c, -mc));
        const float a1 = fast_exp2(fmaf(bf_lo(v.y), c, -mc)) + fast_exp2(fmaf(bf_hi(v.y), c, -mc));
        const float a2 = fast_exp2(fmaf(bf_lo(v.z), c, -mc)) + fast_exp2(fmaf(bf_hi(v.z), c, -mc));
        const float a3 = fast_exp2(fmaf(bf_lo(v.w), c, -mc)) + fast_exp2(fmaf(bf_hi(v.w), c, -mc));
        return (a0 + a1) + (a2 + a3);
    }
    // the same sum as a pair (x c - mc by packed fma; c2 = (c, c), nmc2 = (-mc, -mc))
    __device__ static __forceinline__ unsigned long long vexp2(const uint4& v, unsigned long long c2,
                                                              unsigned long long nmc2) {
        const unsigned long long e0 = f2_exp2(f2_fma(f2_pack(bf_lo(v.x), bf_hi(v.x)), c2, nmc2));
        const unsigned long long e1 = f2_exp2(f2_fma(f2_pack(bf_lo(v.y), bf_hi(v.y)), c2, nmc2));
        const unsigned long long e2 = f2_exp2(f2_fma(f2_pack(bf_lo(v.z), bf_hi(v.z)), c2, nmc2));
        const unsigned long long e3 = f2_exp2(f2_fma(f2_pack(bf_lo(v.w), bf_hi(v.w)), c2, nmc2));
        return f2_add(f2_add(e0, e1), f2_add(e2, e3));
    }
    // bit i set when element i is >= t (t2: t as a bf16 pair; false for NaN)
    __device__ static __forceinline__ uint32_t ge_bits(const uint4& v, uint32_t t2) {
        const __nv_bfloat162 t = *reinterpret_cast<const __nv_bfloat162*>(&t2);
        auto mk = [&](uint32_t w) { return __hge2_mask(*reinterpret_cast<const __nv_bfloat162*>(&w), t) & 0x00010001u; };
        const uint32_t x = mk(v.x) | (mk(v.y) << 2) | (mk(v.z) << 4) | (mk(v.w) << 6);
        return (x & 0x55u) | ((x >> 15) & 0xAAu);
    }
    // elements [nv, 8) become -inf
    __device__ static __forceinline__ uint4 mask(uint4 v, int nv) {
        auto m = [](uint32_t w, int lo_idx, int nv) -> uint32_t {
            if (lo_idx >= nv) return 0xFF80FF80u;
            if (lo_idx + 1 >= nv) return (w & 0xFFFFu) | 0xFF800000u;
            return w;
        };
        return make_uint4(m(v.x, 0, nv), m(v.y, 2, nv), m(v.z, 4, nv), m(v.w, 6, nv));
    }
};
template <> struct Vec<0> {
    __device__ static __forceinline__ float vmax(const uint4& v) {
        return fmaxf(fmaxf(__uint_as_float(v.x), __uint_as_float(v.y)),
                     fmaxf(__uint_as_float(v.z), __uint_as_float(v.w)));
    }
    __device__ static __forceinline__ float vexp(const uint4& v, float c, float mc) {
        const float a0 = fast_exp2(fmaf(__uint_as_float(v.x), c, -mc)) + fast_exp2(fmaf(__uint_as_float(v.y), c, -mc));
        const float a1 = fast_exp2(fmaf(__uint_as_float(v.z), c, -mc)) + fast_exp2(fmaf(__uint_as_float(v.w), c, -mc));
        return a0 + a1;
    }
    __device__ static __forceinline__ unsigned long long vexp2(const uint4& v, unsigned long long c2,
                                                              unsigned long long nmc2) {
        const unsigned long long e0 =
            f2_exp2(f2_fma(f2_pack(__uint_as_float(v.x), __uint_as_float(v.y)), c2, nmc2));
        const unsigned long long e1 =
            f2_exp2(f2_fma(f2_pack(__uint_as_float(v.z), __uint_as_float(v.w)), c2, nmc2));
        return f2_add(e0, e1);
    }
    __device__ static __forceinline__ uint32_t ge_bits(const uint4& v, uint32_t t2) {
        const float t = __uint_as_float(t2);
        return (__uint_as_float(v.x) >= t ? 1u : 0u) | (__uint_as_float(v.y) >= t ? 2u : 0u) |
               (__uint_as_float(v.z) >= t ? 4u : 0u) | (__uint_as_float(v.w) >= t ? 8u : 0u);
    }
    __device__ static __forceinline__ uint4 mask(uint4 v, int nv) {
        const uint32_t ni = 0xFF800000u;
        return make_uint4(nv > 0 ? v.x : ni, nv > 1 ? v.y : ni, nv > 2 ? v.z : ni, nv > 3 ? v.w : ni);
    }
};

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
// block reductions (NW warps, all threads must call; NW = kWarps by default)
// ---------------------------------------------------------------------------
struct BlockScratch {
    int ired[2][kMaxWarps];
    float fred[kMaxWarps];
    float fred2[kMaxWarps];
    unsigned long long ured[kMaxWarps];
    int flag;
};

template <int NW = kWarps>
__device__ __forceinline__ int block_sum_int(int v, BlockScratch& s, int& parity) {
    v = __reduce_add_sync(0xFFFFFFFFu, v);
    int* buf = s.ired[parity];
    parity ^= 1;
    if ((threadIdx.x & 31) == 0) buf[threadIdx.x >> 5] = v;
    __syncthreads();
    int t = 0;
#pragma unroll
    for (int w = 0; w < NW; ++w) t += buf[w];
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

template <int NW = kWarps>
__device__ __forceinline__ unsigned long long block_max_u64(unsigned long long v, BlockScratch& s) {
    v = warp_max_u64(v);
    __syncthreads();
    if ((threadIdx.x & 31) == 0) s.ured[threadIdx.x >> 5] = v;
    __syncthreads();
    unsigned long long t = 0;
#pragma unroll
    for (int w = 0; w < NW; ++w) t = s.ured[w] > t ? s.ured[w] : t;
    return t;
}

template <int NW = kWarps>
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
    for (int w = 0; w < NW; ++w) t = want_or ? (t | s.ured[w]) : (t & s.ured[w]);
    return t;
}

// block-wide maximum (all threads get it)
template <int NW = kWarps>
__device__ __forceinline__ float block_max_f32(float v, BlockScratch& s) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
    __syncthreads();
    if ((threadIdx.x & 31) == 0) s.fred[threadIdx.x >> 5] = v;
    __syncthreads();
    float m = s.fred[0];
#pragma unroll
    for (int w = 1; w < NW; ++w) m = fmaxf(m, s.fred[w]);
    return m;
}

// ---------------------------------------------------------------------------
// float-float arithmetic (value = hi + lo, ~48 significant bits) in place of
// fp64, whose throughput on this part is a tiny fraction of fp32's.  The
// explicit _rn intrinsics keep the compiler from contracting the error terms.
// ---------------------------------------------------------------------------
struct FF {
    float hi, lo;
};
__device__ __forceinline__ FF ff_two_sum(float a, float b) {
    const float s = __fadd_rn(a, b);
    const float bb = __fsub_rn(s, a);
    const float e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
    return {s, e};
}
__device__ __forceinline__ FF ff_norm(float a, float b) {  // |a| >= |b|
    const float s = __fadd_rn(a, b);
    return {s, __fsub_rn(b, __fsub_rn(s, a))};
}
__device__ __forceinline__ FF ff_add(FF x, FF y) {
    if (!(x.hi > -INFINITY && x.hi < INFINITY) || !(y.hi > -INFINITY && y.hi < INFINITY))
        return {__fadd_rn(x.hi, y.hi), 0.0f};
    const FF s = ff_two_sum(x.hi, y.hi);
    return ff_norm(s.hi, __fadd_rn(s.lo, __fadd_rn(x.lo, y.lo)));
}
__device__ __forceinline__ FF ff_add(FF x, float y) { return ff_add(x, FF{y, 0.0f}); }
__device__ __forceinline__ FF ff_neg(FF x) { return {-x.hi, -x.lo}; }
__device__ __forceinline__ FF ff_shfl_xor(FF x, int o) {
    return {__shfl_xor_sync(0xFFFFFFFFu, x.hi, o), __shfl_xor_sync(0xFFFFFFFFu, x.lo, o)};
}
// a * x exactly enough: (p + e) with e the fma residue
__device__ __forceinline__ FF ff_mul(float a, FF x) {
    const float p = __fmul_rn(a, x.hi);
    const float e = fmaf(a, x.hi, -p);
    return ff_norm(p, fmaf(a, x.lo, e));
}
// log of a positive float-float (first-order correction of logf)
__device__ __forceinline__ FF ff_log(FF x) {
    const float y = logf(x.hi);
    if (!(x.hi > 0.0f) || !(y > -INFINITY && y < INFINITY)) return {y, 0.0f};
    return ff_two_sum(y, __fdiv_rn(x.lo, x.hi));
}
// v / T as float-float: correctly rounded quotient plus the exact fma remainder
__device__ __forceinline__ FF ff_div(float v, float T) {
    const float q = __fdiv_rn(v, T);
    if (!(q > -INFINITY && q < INFINITY)) return {q, 0.0f};
    return {q, __fdiv_rn(fmaf(-q, T, v), T)};
}
// "a <= b" for b a float and a = x (float-float), decided exactly enough
__device__ __forceinline__ bool ff_le(FF x, float b) {
    const float d = __fsub_rn(b, x.hi);
    return d > x.lo || (d == x.lo);
}

// block-wide sum of fp32 values: float-float (compensated) in and across warps
template <int NW = kWarps>
__device__ __forceinline__ FF block_sum_ff(FF v, BlockScratch& s) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = ff_add(v, ff_shfl_xor(v, o));
    __syncthreads();
    if ((threadIdx.x & 31) == 0) {
        s.fred[threadIdx.x >> 5] = v.hi;
        s.fred2[threadIdx.x >> 5] = v.lo;
    }
    __syncthreads();
    FF t{s.fred[0], s.fred2[0]};
#pragma unroll
    for (int w = 1; w < NW; ++w) t = ff_add(t, FF{s.fred[w], s.fred2[w]});
    return t;
}
template <int NW = kWarps>
__device__ __forceinline__ FF block_sum_ff(float v, BlockScratch& s) { return block_sum_ff<NW>(FF{v, 0.0f}, s); }

// ---------------------------------------------------------------------------
// Block reductions with one barrier each: the warp partials go to one of two
// scratch buffers, alternated by the caller's parity bit, so a warp that runs
// ahead into the next reduction never overwrites partials still being read.
// ---------------------------------------------------------------------------
struct Red {
    float f[2][kMaxWarps];
    float g[2][kMaxWarps];
    unsigned long long u[2][kMaxWarps];
    int i[2][kMaxWarps];
};

template <int NW = kWarps>
__device__ __forceinline__ float red_max_f32(float v, Red& r, int& par) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
    float* buf = r.f[par];
    par ^= 1;
    if ((threadIdx.x & 31) == 0) buf[threadIdx.x >> 5] = v;
    __syncthreads();
    float m = buf[0];
#pragma unroll
    for (int w = 1; w < NW; ++w) m = fmaxf(m, buf[w]);
    return m;
}

template <int NW = kWarps>
__device__ __forceinline__ FF red_sum_ff(FF v, Red& r, int& par) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = ff_add(v, ff_shfl_xor(v, o));
    float* bh = r.f[par];
    float* bl = r.g[par];
    par ^= 1;
    if ((threadIdx.x & 31) == 0) {
        bh[threadIdx.x >> 5] = v.hi;
        bl[threadIdx.x >> 5] = v.lo;
    }
    __syncthreads();
    // the warp partials combined by a shuffle tree in every warp (log2 NW
    // dependent steps instead of NW), then taken from lane 0: all threads agree
    const int lane = threadIdx.x & 31;
    FF t = lane < NW ? FF{bh[lane], bl[lane]} : FF{0.0f, 0.0f};
#pragma unroll
    for (int o = NW / 2; o > 0; o >>= 1) t = ff_add(t, ff_shfl_xor(t, o));
    return FF{__shfl_sync(0xFFFFFFFFu, t.hi, 0), __shfl_sync(0xFFFFFFFFu, t.lo, 0)};
}

// Block sum (float-float) and maximum (u64) in one barrier: both partials of
// every warp go to the scratch at once, then the same shuffle trees as
// red_sum_ff and red_max_u64 combine them in every warp.
template <int NW = kWarps>
__device__ __forceinline__ void red_sum_ff_max_u64(FF v, unsigned long long k, Red& r, int& par, FF& sum,
                                                   unsigned long long& mx) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        v = ff_add(v, ff_shfl_xor(v, o));
        const unsigned long long y = __shfl_xor_sync(0xFFFFFFFFu, k, o);
        k = y > k ? y : k;
    }
    float* bh = r.f[par];
    float* bl = r.g[par];
    unsigned long long* bu = r.u[par];
    par ^= 1;
    if ((threadIdx.x & 31) == 0) {
        bh[threadIdx.x >> 5] = v.hi;
        bl[threadIdx.x >> 5] = v.lo;
        bu[threadIdx.x >> 5] = k;
    }
    __syncthreads();
    const int lane = threadIdx.x & 31;
    FF t = lane < NW ? FF{bh[lane], bl[lane]} : FF{0.0f, 0.0f};
    unsigned long long q = lane < NW ? bu[lane] : 0ull;
#pragma unroll
    for (int o = NW / 2; o > 0; o >>= 1) {
        t = ff_add(t, ff_shfl_xor(t, o));
        const unsigned long long y = __shfl_xor_sync(0xFFFFFFFFu, q, o);
        q = y > q ? y : q;
    }
    sum = FF{__shfl_sync(0xFFFFFFFFu, t.hi, 0), __shfl_sync(0xFFFFFFFFu, t.lo, 0)};
    mx = __shfl_sync(0xFFFFFFFFu, q, 0);
}

template <int NW = kWarps>
__device__ __forceinline__ unsigned long long red_max_u64(unsigned long long v, Red& r, int& par) {
    v = warp_max_u64(v);
    unsigned long long* buf = r.u[par];
    par ^= 1;
    if ((threadIdx.x & 31) == 0) buf[threadIdx.x >> 5] = v;
    __syncthreads();
    unsigned long long t = (threadIdx.x & 31) < NW ? buf[threadIdx.x & 31] : 0ull;
#pragma unroll
    for (int o = NW / 2; o > 0; o >>= 1) {
        const unsigned long long y = __shfl_xor_sync(0xFFFFFFFFu, t, o);
        t = y > t ? y : t;
    }
    return __shfl_sync(0xFFFFFFFFu, t, 0);
}

template <int NW = kWarps>
__device__ __forceinline__ int red_sum_int(int v, Red& r, int& par) {
    v = __reduce_add_sync(0xFFFFFFFFu, v);
    int* buf = r.i[par];
    par ^= 1;
    if ((threadIdx.x & 31) == 0) buf[threadIdx.x >> 5] = v;
    __syncthreads();
    int t = 0;
#pragma unroll
    for (int w = 0; w < NW; ++w) t += buf[w];
    return t;
}

// exclusive prefix sum in thread order; total in `total`
template <int NW = kWarps>
__device__ __forceinline__ int red_scan(int v, int& total, Red& r, int& par) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xFFFFFFFFu, x, o);
        if (lane >= o) x += y;
    }
    int* buf = r.i[par];
    par ^= 1;
    if (lane == 31) buf[warp] = x;
    __syncthreads();
    int before = 0;
    total = 0;
#pragma unroll
    for (int w = 0; w < NW; ++w) {
        before += (w < warp) ? buf[w] : 0;
        total += buf[w];
    }
    return before + x - v;
}

// Partition sum of a block: every thread holds (m, s) = (its maximum, sum of
// 2^((x - m) c) over its values; m = -inf when it has none).  Returns
// M = max over the block and the sum rescaled to M as float-float.
template <int NW = kWarps>
__device__ __forceinline__ FF red_partition(float m, float s, float c, float& M, Red& r, int& par) {
    // in the warp: common maximum first, each sum rescaled to it once, then a
    // plain fp32 tree (5 levels: relative error below 5 * 2^-24)
    float mw = m;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mw = fmaxf(mw, __shfl_xor_sync(0xFFFFFFFFu, mw, o));
    float sw = (m == -INFINITY) ? 0.0f : s * fast_exp2((m - mw) * c);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sw += __shfl_xor_sync(0xFFFFFFFFu, sw, o);
    m = mw;
    FF v{sw, 0.0f};
    float* bm = r.f[par];
    float* bh = r.g[par];
    unsigned long long* bl = r.u[par];
    par ^= 1;
    if ((threadIdx.x & 31) == 0) {
        bm[threadIdx.x >> 5] = m;
        bh[threadIdx.x >> 5] = v.hi;
        bl[threadIdx.x >> 5] = (unsigned long long)__float_as_uint(v.lo);
    }
    __syncthreads();
    // the same pairwise rescale-and-add over the warp partials, as a shuffle
    // tree in every warp, taken from lane 0
    const int lane = threadIdx.x & 31;
    m = lane < NW ? bm[lane] : -INFINITY;
    v = lane < NW ? FF{bh[lane], __uint_as_float((uint32_t)bl[lane])} : FF{0.0f, 0.0f};
#pragma unroll
    for (int o = NW / 2; o > 0; o >>= 1) {
        const float m2 = __shfl_xor_sync(0xFFFFFFFFu, m, o);
        const FF v2 = ff_shfl_xor(v, o);
        const float mm = fmaxf(m, m2);
        const FF a = (m == -INFINITY) ? FF{0.0f, 0.0f} : ff_mul(fast_exp2((m - mm) * c), v);
        const FF b = (m2 == -INFINITY) ? FF{0.0f, 0.0f} : ff_mul(fast_exp2((m2 - mm) * c), v2);
        v = ff_add(a, b);
        m = mm;
    }
    M = __shfl_sync(0xFFFFFFFFu, m, 0);
    return FF{__shfl_sync(0xFFFFFFFFu, v.hi, 0), __shfl_sync(0xFFFFFFFFu, v.lo, 0)};
}

// exp(l / T - c) for an fp32 logit l and a float-float constant c, to a few
// fp32 ulps: l / T = tau + rem / T exactly (tau correctly rounded).
__device__ __forceinline__ float exp_scaled_minus(float l, float T, FF c) {
    const FF x = ff_div(l, T);
    if (!(x.hi > -INFINITY && x.hi < INFINITY)) return expf(x.hi - c.hi);
    const float d = __fsub_rn(x.hi, c.hi) + (x.lo - c.lo);
    return expf(d);
}

// ---------------------------------------------------------------------------
// Selection: threshold T with count(keys >= T) == k for k <= n distinct 64-bit
// keys spread over the block (for keys with repeats: the k-th largest key).
// Bits shared by every key are taken from their AND at once; the rest is a
// radix select on 8-bit digits, most significant first: a shared histogram per
// digit, a block scan over the digits from the top, stop as soon as the keys
// at or above the current prefix number exactly k.  get(i), i in [0, n)
// visited as i = tid + j * NT (NT threads, NT >= kRadixBins), returns a key, or 0 for "no key".
// ---------------------------------------------------------------------------
constexpr int kRadixBins = 256;

struct RadixScratch {
    unsigned long long red_and[kMaxWarps], red_or[kMaxWarps];
    int wsum[kMaxWarps];
    int digit, above;
};

template <int NT = kThreads, class Get>
__device__ unsigned long long block_radix_threshold(Get get, int n, int k, unsigned* hist, RadixScratch& rs) {
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    // common leading bits
    unsigned long long a_and = ~0ull, a_or = 0ull;
    for (int i = tid; i < n; i += NT) {
        const unsigned long long x = get(i);
        if (x) { a_and &= x; a_or |= x; }
    }
    {
        unsigned lo_a = __reduce_and_sync(0xFFFFFFFFu, (unsigned)a_and), hi_a = __reduce_and_sync(0xFFFFFFFFu, (unsigned)(a_and >> 32));
        unsigned lo_o = __reduce_or_sync(0xFFFFFFFFu, (unsigned)a_or), hi_o = __reduce_or_sync(0xFFFFFFFFu, (unsigned)(a_or >> 32));
        if (lane == 0) {
            rs.red_and[warp] = ((unsigned long long)hi_a << 32) | lo_a;
            rs.red_or[warp] = ((unsigned long long)hi_o << 32) | lo_o;
        }
        __syncthreads();
        a_and = ~0ull;
        a_or = 0ull;
#pragma unroll
        for (int w = 0; w < NT / 32; ++w) { a_and &= rs.red_and[w]; a_or |= rs.red_or[w]; }
    }
    const unsigned long long diff = a_and ^ a_or;
    if (diff == 0ull) {  // all keys equal
        __syncthreads();
        return a_and;
    }
    int top = 64 - __clzll((long long)diff);  // bits >= top are common to every key
    unsigned long long prefix = (top >= 64) ? 0ull : (a_and >> top) << top;
    int above = 0;
    while (top > 0) {
        const int bits = top >= 8 ? 8 : top;
        const int shift = top - bits;
        const unsigned mask = (1u << bits) - 1u;
        if (tid < kRadixBins) hist[tid] = 0u;
        if (tid == 0) rs.digit = -1;
        __syncthreads();
        for (int i = tid; i < n; i += NT) {
            const unsigned long long x = get(i);
            if (x == 0ull) continue;
            if (top < 64 && (x >> top) != (prefix >> top)) continue;
            atomicAdd(&hist[(unsigned)(x >> shift) & mask], 1u);
        }
        __syncthreads();
        // thread t owns digit 255 - t (descending order of digits)
        const int d = kRadixBins - 1 - tid;
        const int h = tid < kRadixBins ? (int)hist[d] : 0;
        int incl = h;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
            if (lane >= o) incl += y;
        }
        if (lane == 31) rs.wsum[warp] = incl;
        __syncthreads();
        int before = above + incl - h;
#pragma unroll
        for (int w = 0; w < NT / 32; ++w) before += (w < warp) ? rs.wsum[w] : 0;
        if (h > 0 && before < k && before + h >= k) {
            rs.digit = d;
            rs.above = before;
        }
        __syncthreads();
        const int dd = rs.digit;
        if (dd < 0 || dd >= kRadixBins) {  // fewer keys than k (broken input): keep every key
            __syncthreads();
            return 1ull;
        }
        above = rs.above;
        prefix |= (unsigned long long)dd << shift;
        const bool exact = above + (int)hist[dd] == k;
        __syncthreads();  // everybody has read rs and hist before they change
        top = shift;
        if (exact) break;
    }
    return prefix;
}

// ---------------------------------------------------------------------------
// k-th largest of up to N values per lane across one warp (0 = "no value"):
// built bit by bit from the most significant bit on, visiting only the bits in
// which the values differ (bits common to all of them come from their AND).
// Returns 0 when the warp holds fewer than k values.  All lanes get the result.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t warp_and_u32(uint32_t x) { return __reduce_and_sync(0xFFFFFFFFu, x); }
__device__ __forceinline__ uint32_t warp_or_u32(uint32_t x) { return __reduce_or_sync(0xFFFFFFFFu, x); }
__device__ __forceinline__ unsigned long long warp_and(unsigned long long x) {
    return ((unsigned long long)warp_and_u32((uint32_t)(x >> 32)) << 32) | warp_and_u32((uint32_t)x);
}
__device__ __forceinline__ unsigned long long warp_or(unsigned long long x) {
    return ((unsigned long long)warp_or_u32((uint32_t)(x >> 32)) << 32) | warp_or_u32((uint32_t)x);
}
__device__ __forceinline__ uint32_t warp_and(uint32_t x) { return warp_and_u32(x); }
__device__ __forceinline__ uint32_t warp_or(uint32_t x) { return warp_or_u32(x); }

template <int N, class T>
__device__ __forceinline__ T warp_kth_largest_of(const T (&x)[N], int k) {
    T a = ~T(0), o = T(0);
    int c = 0;
#pragma unroll
    for (int i = 0; i < N; ++i)
        if (x[i]) {
            a &= x[i];
            o |= x[i];
            ++c;
        }
    c = __reduce_add_sync(0xFFFFFFFFu, c);
    if (c < k) return T(0);
    a = warp_and(a);
    o = warp_or(o);
    T prefix = a;
    for (T diff = a ^ o; diff;) {
        const int bit = (int)(sizeof(T) * 8 - 1) - (sizeof(T) == 8 ? __clzll((long long)diff) : __clz((int)diff));
        const T b = T(1) << bit;
        diff ^= b;
        const T cand = prefix | b;
        int q = 0;
#pragma unroll
        for (int i = 0; i < N; ++i) q += (x[i] >= cand) ? 1 : 0;
        if (__reduce_add_sync(0xFFFFFFFFu, q) >= k) prefix = cand;
    }
    return prefix;
}

// ---------------------------------------------------------------------------
// Block-wide k-th largest of n distinct nonzero 64-bit keys (get(i) == 0 means
// "no key"; i visited as tid + j * NT, NT >= kRadixBins threads), 1 <= k <= number of keys.  The
// returned threshold T has exactly k keys >= T.  Rounds over the keys still in
// play ("live": equal to the prefix found so far above bit `top`): bits common
// to every live key are taken from their AND at once, the next 8 differing
// bits are counted in a shared histogram and scanned from the top; a round
// ends early when the keys at or above the prefix number exactly k, and a tie
// class of at most 32 keys is finished by one warp ranking it.
// ---------------------------------------------------------------------------
struct SelScratch {
    unsigned long long red_and[kMaxWarps], red_or[kMaxWarps];
    int wsum[kMaxWarps];
    int digit, above, tie_n;
    unsigned long long result;
    unsigned long long tie[32];
};

template <int NT = kThreads, class Get>
__device__ unsigned long long block_kth_key(Get get, int n, int k, unsigned* hist, SelScratch& ss) {
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    unsigned long long prefix = 0ull;
    int top = 64, above = 0;
    auto live = [&](unsigned long long x) -> bool {
        return x != 0ull && (top >= 64 || (x >> top) == (prefix >> top));
    };
    for (;;) {
        // common bits of the live keys; the histogram is cleared meanwhile
        unsigned long long a_and = ~0ull, a_or = 0ull;
        int nl = 0;
        for (int i = tid; i < n; i += NT) {
            const unsigned long long x = get(i);
            if (live(x)) {
                a_and &= x;
                a_or |= x;
                ++nl;
            }
        }
        a_and = warp_and(a_and);
        a_or = warp_or(a_or);
        nl = __reduce_add_sync(0xFFFFFFFFu, nl);
        if (lane == 0) {
            ss.red_and[warp] = a_and;
            ss.red_or[warp] = a_or;
            ss.wsum[warp] = nl;
        }
        if (tid < kRadixBins) hist[tid] = 0u;
        if (tid == 0) ss.digit = -1;
        __syncthreads();
        a_and = ~0ull;
        a_or = 0ull;
        nl = 0;
#pragma unroll
        for (int w = 0; w < NT / 32; ++w) {
            a_and &= ss.red_and[w];
            a_or |= ss.red_or[w];
            nl += ss.wsum[w];
        }
        if (nl == 0 || above + nl < k) {  // fewer keys than k (broken input): keep every key
            __syncthreads();
            return 1ull;
        }
        const unsigned long long diff = a_and ^ a_or;
        if (diff == 0ull) {  // a single live key: the k-th
            __syncthreads();
            return a_and;
        }
        top = 64 - __clzll((long long)diff);
        prefix = (top >= 64) ? 0ull : (a_and >> top) << top;
        const int bits = top >= 8 ? 8 : top;
        const int shift = top - bits;
        const unsigned mask = (1u << bits) - 1u;
        for (int i = tid; i < n; i += NT) {
            const unsigned long long x = get(i);
            if (live(x)) atomicAdd(&hist[(unsigned)(x >> shift) & mask], 1u);
        }
        __syncthreads();
        // thread t owns digit 255 - t: digits in descending order
        const int d = kRadixBins - 1 - tid;
        const int h = tid < kRadixBins ? (int)hist[d] : 0;
        int incl = h;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xFFFFFFFFu, incl, o);
            if (lane >= o) incl += y;
        }
        if (lane == 31) ss.wsum[warp] = incl;
        __syncthreads();
        int before = above + incl - h;
#pragma unroll
        for (int w = 0; w < NT / 32; ++w) before += (w < warp) ? ss.wsum[w] : 0;
        if (h > 0 && before < k && before + h >= k) {
            ss.digit = d;
            ss.above = before;
            ss.tie_n = 0;
        }
        __syncthreads();
        const int dd = ss.digit;
        if (dd < 0) {  // cannot happen when the keys number at least k
            __syncthreads();
            return 1ull;
        }
        above = ss.above;
        const int cnt = (int)hist[dd];
        prefix |= (unsigned long long)dd << shift;
        top = shift;
        if (above + cnt == k) {
            __syncthreads();
            return prefix;
        }
        if (cnt <= 32) {  // finish the tie class in one warp
            for (int i = tid; i < n; i += NT) {
                const unsigned long long x = get(i);
                if (live(x)) ss.tie[atomicAdd(&ss.tie_n, 1)] = x;
            }
            __syncthreads();
            if (warp == 0) {
                const unsigned long long x = lane < cnt ? ss.tie[lane] : 0ull;
                int rank = 0;
#pragma unroll
                for (int j = 0; j < 32; ++j) rank += (__shfl_sync(0xFFFFFFFFu, x, j) > x) ? 1 : 0;
                if (x && rank == k - above - 1) ss.result = x;
            }
            __syncthreads();
            return ss.result;
        }
        __syncthreads();  // hist and ss read by everyone before the next round
    }
}

// exclusive prefix sum over the block (in thread order)
template <int NW = kWarps>
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
    for (int w = 0; w < NW; ++w) {
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

// numbering helpers (see rheo.h); gen ids < 2^14, so 32-bit arithmetic
__device__ __forceinline__ int depth_base(int K, int d) { return d == 1 ? 1 : 1 + (K + 1) + (d - 2) * K * (K + 1); }
__device__ __forceinline__ int slot_of(int K, int g) { return g <= K + 1 ? g - 1 : (g - (K + 2)) % (K + 1); }
__device__ __forceinline__ int parent_expansion_of(int K, int g) {
    if (g <= K + 1) return 0;
    const int w = g - (K + 2), per = K * (K + 1);
    return 1 + (w / per) * K + (w % per) / (K + 1);
}
__device__ __forceinline__ int depth_of(int K, int g) {
    if (g == 0) return 0;
    if (g <= K + 1) return 1;
    return 2 + (g - (K + 2)) / (K * (K + 1));
}

}  // namespace rheo
