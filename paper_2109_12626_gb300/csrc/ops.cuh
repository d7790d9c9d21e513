// ops.cuh -- the (.) functors of the library and the memory units the
// kernels move.  A functor combines a (.) b with a the LOWER-ranked operand
// (the problem statement of Sec. 1 keeps rank order for a non-commutative
// operator).
//
// Two unit kinds carry data through every kernel:
//   Vec  16 bytes = 4 int32 / 4 float32 / 1 matrix, one 128-bit access;
//        needs every rank buffer 16-byte aligned.
//   One  one element, moved with 4-byte accesses; used for the ragged tail
//        of a vectorised problem and for buffers that are only 4-byte
//        aligned.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace dpdr {

struct SumI32 {
    static constexpr int kEpv = 4;  // elements per 16-byte vector
    static constexpr int kEsize = 4;
    __device__ __forceinline__ static uint4 vec(uint4 a, uint4 b)
    {
        return make_uint4(a.x + b.x, a.y + b.y, a.z + b.z, a.w + b.w);
    }
    // one element, as raw 32-bit words (w[0] used)
    __device__ __forceinline__ static void one(const uint32_t* a,
                                               const uint32_t* b, uint32_t* o)
    {
        o[0] = a[0] + b[0];
    }
};

struct SumF32 {
    static constexpr int kEpv = 4;
    static constexpr int kEsize = 4;
    __device__ __forceinline__ static uint32_t add(uint32_t a, uint32_t b)
    {
        // one IEEE single add, round to nearest even, never contracted
        return __float_as_uint(__fadd_rn(__uint_as_float(a), __uint_as_float(b)));
    }
    __device__ __forceinline__ static uint4 vec(uint4 a, uint4 b)
    {
        return make_uint4(add(a.x, b.x), add(a.y, b.y), add(a.z, b.z), add(a.w, b.w));
    }
    __device__ __forceinline__ static void one(const uint32_t* a,
                                               const uint32_t* b, uint32_t* o)
    {
        o[0] = add(a[0], b[0]);
    }
};

// 2x2 matrices mod 2^32, row-major (x y / z w): [a0 a1; a2 a3] [b0 b1; b2 b3]
struct MatU32 {
    static constexpr int kEpv = 1;
    static constexpr int kEsize = 16;
    __device__ __forceinline__ static uint4 vec(uint4 a, uint4 b)
    {
        return make_uint4(a.x * b.x + a.y * b.z, a.x * b.y + a.y * b.w,
                          a.z * b.x + a.w * b.z, a.z * b.y + a.w * b.w);
    }
    __device__ __forceinline__ static void one(const uint32_t* a,
                                               const uint32_t* b, uint32_t* o)
    {
        const uint4 r = vec(make_uint4(a[0], a[1], a[2], a[3]),
                            make_uint4(b[0], b[1], b[2], b[3]));
        o[0] = r.x;
        o[1] = r.y;
        o[2] = r.z;
        o[3] = r.w;
    }
};

// 2x2 float32 matrices, row-major; every entry is two rounded products and
// one rounded sum (never contracted into an FMA), so the result is defined
// by the bracketing alone: non-commutative, and non-associative in rounding.
struct MatF32 {
    static constexpr int kEpv = 1;
    static constexpr int kEsize = 16;
    __device__ __forceinline__ static uint32_t dot(uint32_t a, uint32_t b, uint32_t c, uint32_t d)
    {
        const float u = __fmul_rn(__uint_as_float(a), __uint_as_float(b));
        const float v = __fmul_rn(__uint_as_float(c), __uint_as_float(d));
        return __float_as_uint(__fadd_rn(u, v));
    }
    __device__ __forceinline__ static uint4 vec(uint4 a, uint4 b)
    {
        return make_uint4(dot(a.x, b.x, a.y, b.z), dot(a.x, b.y, a.y, b.w),
                          dot(a.z, b.x, a.w, b.z), dot(a.z, b.y, a.w, b.w));
    }
    __device__ __forceinline__ static void one(const uint32_t* a, const uint32_t* b, uint32_t* o)
    {
        const uint4 r = vec(make_uint4(a[0], a[1], a[2], a[3]), make_uint4(b[0], b[1], b[2], b[3]));
        o[0] = r.x;
        o[1] = r.y;
        o[2] = r.z;
        o[3] = r.w;
    }
};

__device__ __forceinline__ int64_t lmin(int64_t a, int64_t b) { return a < b ? a : b; }

// ------------------------------------------------------------ memory units
// Streaming hints: inputs are read once (evict-first), outputs written once.
__device__ __forceinline__ uint4 ld_stream(const void* p)
{
    return __ldcs(reinterpret_cast<const uint4*>(p));
}
__device__ __forceinline__ void st_stream(void* p, uint4 v)
{
    __stcs(reinterpret_cast<uint4*>(p), v);
}
// L2-coherent accesses for data another CTA of the same kernel produced
__device__ __forceinline__ uint4 ld_l2(const void* p)
{
    return __ldcg(reinterpret_cast<const uint4*>(p));
}
__device__ __forceinline__ void st_l2(void* p, uint4 v)
{
    __stcg(reinterpret_cast<uint4*>(p), v);
}
__device__ __forceinline__ uint32_t ld_l2_u32(const void* p)
{
    return __ldcg(reinterpret_cast<const unsigned int*>(p));
}
__device__ __forceinline__ void st_l2_u32(void* p, uint32_t v)
{
    __stcg(reinterpret_cast<unsigned int*>(p), v);
}

// One element of Op held in registers: 1 word (int32/float32) or 4 (matrix)
template <class Op>
struct Elem {
    static constexpr int kWords = Op::kEsize / 4;
    uint32_t w[kWords];
};

template <class Op>
__device__ __forceinline__ Elem<Op> ld_one_stream(const char* p)
{
    Elem<Op> e;
#pragma unroll
    for (int k = 0; k < Elem<Op>::kWords; k++)
        e.w[k] = __ldcs(reinterpret_cast<const unsigned int*>(p) + k);
    return e;
}
template <class Op>
__device__ __forceinline__ void st_one_stream(char* p, const Elem<Op>& e)
{
#pragma unroll
    for (int k = 0; k < Elem<Op>::kWords; k++)
        __stcs(reinterpret_cast<unsigned int*>(p) + k, e.w[k]);
}
template <class Op>
__device__ __forceinline__ Elem<Op> ld_one_l2(const char* p)
{
    Elem<Op> e;
#pragma unroll
    for (int k = 0; k < Elem<Op>::kWords; k++)
        e.w[k] = ld_l2_u32(p + 4 * k);
    return e;
}
template <class Op>
__device__ __forceinline__ void st_one_l2(char* p, const Elem<Op>& e)
{
#pragma unroll
    for (int k = 0; k < Elem<Op>::kWords; k++) st_l2_u32(p + 4 * k, e.w[k]);
}
template <class Op>
__device__ __forceinline__ Elem<Op> comb(const Elem<Op>& a, const Elem<Op>& b)
{
    Elem<Op> o;
    Op::one(a.w, b.w, o.w);
    return o;
}

}  // namespace dpdr
