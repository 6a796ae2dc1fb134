// haar.cu -- one level of the 2-D Haar kernel bank of the T-DVAE (Sec. 2.3 DWT-Enhanced
// Architecture) and its inverse, per channel, stride 2, orthonormal:
//   LL = (a+b+c+d)/2, HL = (a-b+c-d)/2, LH = (a+b-c-d)/2, HH = (a-b-c+d)/2
// for the window a = x[2i][2j], b = x[2i][2j+1], c = x[2i+1][2j], d = x[2i+1][2j+1]; the
// inverse is the transpose. HBM-bound: a unit is 16 bytes of each of the two
// input rows (one vector load each), which make 8 bytes of each band; a full grid of units (no
// persistent loop), 32-bit index arithmetic where the unit count allows. fp32 arithmetic, bf16
// or fp32 in and out. Subband-major output: [nb][C][H/2][W/2] per image.
#include <algorithm>

#include "common.cuh"

namespace ssba {

namespace {

// Lane packing of a 16-byte row segment (2V elements) and an 8-byte band segment (V elements).
template <typename T>
struct Lanes;
template <>
struct Lanes<float> {
    static constexpr int V = 2;
    __device__ static void unpack16(const uint4& u, float (&f)[4])
    {
        f[0] = __uint_as_float(u.x);
        f[1] = __uint_as_float(u.y);
        f[2] = __uint_as_float(u.z);
        f[3] = __uint_as_float(u.w);
    }
    __device__ static void unpack8(const uint2& u, float (&f)[2])
    {
        f[0] = __uint_as_float(u.x);
        f[1] = __uint_as_float(u.y);
    }
    __device__ static uint2 pack8(const float (&f)[2]) { return make_uint2(__float_as_uint(f[0]), __float_as_uint(f[1])); }
    __device__ static uint4 pack16(const float (&f)[4])
    {
        return make_uint4(__float_as_uint(f[0]), __float_as_uint(f[1]), __float_as_uint(f[2]), __float_as_uint(f[3]));
    }
};
template <>
struct Lanes<__nv_bfloat16> {
    static constexpr int V = 4;
    __device__ static float2 lo_hi(uint32_t w) { return __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w)); }
    __device__ static uint32_t pk(float a, float b)
    {
        __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
        return *reinterpret_cast<uint32_t*>(&h);
    }
    __device__ static void unpack16(const uint4& u, float (&f)[8])
    {
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const float2 p = lo_hi(w[k]);
            f[2 * k] = p.x;
            f[2 * k + 1] = p.y;
        }
    }
    __device__ static void unpack8(const uint2& u, float (&f)[4])
    {
        const float2 a = lo_hi(u.x), b = lo_hi(u.y);
        f[0] = a.x;
        f[1] = a.y;
        f[2] = b.x;
        f[3] = b.y;
    }
    __device__ static uint2 pack8(const float (&f)[4]) { return make_uint2(pk(f[0], f[1]), pk(f[2], f[3])); }
    __device__ static uint4 pack16(const float (&f)[8])
    {
        return make_uint4(pk(f[0], f[1]), pk(f[2], f[3]), pk(f[4], f[5]), pk(f[6], f[7]));
    }
};

template <bool kStream, typename V>
__device__ __forceinline__ V ld(const V* p)
{
    if constexpr (kStream)
        return __ldcs(p);
    else
        return __ldg(p);
}
template <bool kStream, typename V>
__device__ __forceinline__ void st(V* p, const V& v)
{
    if constexpr (kStream)
        __stcs(p, v);
    else
        *p = v;
}

__device__ __forceinline__ float ldf(const float* p) { return *p; }
__device__ __forceinline__ float ldf(const __nv_bfloat16* p) { return __bfloat162float(*p); }
__device__ __forceinline__ void stf(float* p, float v) { *p = v; }
__device__ __forceinline__ void stf(__nv_bfloat16* p, float v) { *p = __float2bfloat16_rn(v); }

// Vector forward transform (W a multiple of 2V): unit u = (image*channel, output row i,
// segment jv of V output columns); U units per thread, all loads issued before any store.
template <typename T, typename I, int U, bool kStream, int NB>
__global__ void __launch_bounds__(256) ssba_haar_dwt_kernel(const T* __restrict__ x, T* __restrict__ y, I units,
                                                            int C, int H, int W)
{
    constexpr int V = Lanes<T>::V;
    const I h2 = H / 2, w2 = W / 2, wv = W / (2 * V);
    const size_t plane = (size_t)C * h2 * w2;
    for (I base = (I)blockIdx.x * blockDim.x * U + threadIdx.x; base < units; base += (I)gridDim.x * blockDim.x * U) {
        uint4 ra[U], rb[U];
        size_t dst[U];
#pragma unroll
        for (int k = 0; k < U; ++k) {
            const I u = base + (I)k * blockDim.x;
            if (u < units) {
                const I jv = u % wv, t = u / wv, i = t % h2, nc = t / h2, n = nc / C, c = nc - n * C;
                const T* r0 = x + ((size_t)nc * H + 2 * i) * W + 2 * V * jv;
                ra[k] = ld<kStream>(reinterpret_cast<const uint4*>(r0));
                rb[k] = ld<kStream>(reinterpret_cast<const uint4*>(r0 + W));
                dst[k] = ((size_t)n * NB * C + c) * h2 * w2 + (size_t)i * w2 + V * jv;
            }
        }
#pragma unroll
        for (int k = 0; k < U; ++k) {
            if (base + (I)k * blockDim.x < units) {
                float a[2 * V], b[2 * V], band[4][V];
                Lanes<T>::unpack16(ra[k], a);
                Lanes<T>::unpack16(rb[k], b);
#pragma unroll
                for (int e = 0; e < V; ++e) {  // window (a[2e] a[2e+1] / b[2e] b[2e+1])
                    const float p = a[2 * e], q = a[2 * e + 1], r = b[2 * e], w = b[2 * e + 1];
                    band[0][e] = (p + q + r + w) * 0.5f;
                    band[1][e] = (p - q + r - w) * 0.5f;
                    band[2][e] = (p + q - r - w) * 0.5f;
                    band[3][e] = (p - q - r + w) * 0.5f;
                }
#pragma unroll
                for (int s = 0; s < 4; ++s)
                    if (s < NB) st<kStream>(reinterpret_cast<uint2*>(y + dst[k] + s * plane), Lanes<T>::pack8(band[s]));
            }
        }
    }
}

// Scalar forward transform for any even W; unit = (image*channel, output row, output column).
template <typename T>
__global__ void __launch_bounds__(256) ssba_haar_dwt_scalar_kernel(const T* __restrict__ x, T* __restrict__ y, int NC,
                                                                   int C, int H, int W, int nb)
{
    const int h2 = H / 2, w2 = W / 2;
    const long long units = (long long)NC * h2 * w2;
    for (long long u = blockIdx.x * (long long)blockDim.x + threadIdx.x; u < units;
         u += (long long)gridDim.x * blockDim.x) {
        const int j = (int)(u % w2);
        const long long t = u / w2;
        const int i = (int)(t % h2);
        const int nc = (int)(t / h2);
        const T* r0 = x + ((size_t)nc * H + 2 * i) * W + 2 * j;
        const float a = ldf(r0), b = ldf(r0 + 1), c_ = ldf(r0 + W), d = ldf(r0 + W + 1);
        const float band[4] = {(a + b + c_ + d) * 0.5f, (a - b + c_ - d) * 0.5f, (a + b - c_ - d) * 0.5f,
                               (a - b - c_ + d) * 0.5f};
        const int n = nc / C, c = nc - n * C;
#pragma unroll
        for (int s = 0; s < 4; ++s)
            if (s < nb) stf(y + (((size_t)n * nb + s) * C + c) * h2 * w2 + (size_t)i * w2 + j, band[s]);
    }
}

// Vector inverse transform (W a multiple of 2V): V values of each band make 2V columns of
// both output rows; the HH band is zero when nb == 3.
template <typename T, typename I, int U, bool kStream, int NB>
__global__ void __launch_bounds__(256) ssba_haar_iwt_kernel(const T* __restrict__ y, T* __restrict__ x, I units,
                                                            int C, int H, int W)
{
    constexpr int V = Lanes<T>::V;
    const I h2 = H / 2, w2 = W / 2, wv = W / (2 * V);
    const size_t plane = (size_t)C * h2 * w2;
    for (I base = (I)blockIdx.x * blockDim.x * U + threadIdx.x; base < units; base += (I)gridDim.x * blockDim.x * U) {
        uint2 rv[U][4];
        size_t dst[U];
#pragma unroll
        for (int k = 0; k < U; ++k) {
            const I u = base + (I)k * blockDim.x;
            if (u < units) {
                const I jv = u % wv, t = u / wv, i = t % h2, nc = t / h2, n = nc / C, c = nc - n * C;
                const T* src = y + ((size_t)n * NB * C + c) * h2 * w2 + (size_t)i * w2 + V * jv;
#pragma unroll
                for (int s = 0; s < 4; ++s)
                    rv[k][s] = s < NB ? ld<kStream>(reinterpret_cast<const uint2*>(src + s * plane)) : make_uint2(0u, 0u);
                dst[k] = ((size_t)nc * H + 2 * i) * W + 2 * V * jv;
            }
        }
#pragma unroll
        for (int k = 0; k < U; ++k) {
            if (base + (I)k * blockDim.x < units) {
                float v[4][V], top[2 * V], bot[2 * V];
#pragma unroll
                for (int s = 0; s < 4; ++s) Lanes<T>::unpack8(rv[k][s], v[s]);
#pragma unroll
                for (int e = 0; e < V; ++e) {
                    const float LL = v[0][e], HL = v[1][e], LH = v[2][e], HH = v[3][e];
                    top[2 * e] = (LL + HL + LH + HH) * 0.5f;
                    top[2 * e + 1] = (LL - HL + LH - HH) * 0.5f;
                    bot[2 * e] = (LL + HL - LH - HH) * 0.5f;
                    bot[2 * e + 1] = (LL - HL - LH + HH) * 0.5f;
                }
                st<kStream>(reinterpret_cast<uint4*>(x + dst[k]), Lanes<T>::pack16(top));
                st<kStream>(reinterpret_cast<uint4*>(x + dst[k] + W), Lanes<T>::pack16(bot));
            }
        }
    }
}

template <typename T>
__global__ void __launch_bounds__(256) ssba_haar_iwt_scalar_kernel(const T* __restrict__ y, T* __restrict__ x, int NC,
                                                                   int C, int H, int W, int nb)
{
    const int h2 = H / 2, w2 = W / 2;
    const long long units = (long long)NC * h2 * w2;
    for (long long u = blockIdx.x * (long long)blockDim.x + threadIdx.x; u < units;
         u += (long long)gridDim.x * blockDim.x) {
        const int j = (int)(u % w2);
        const long long t = u / w2;
        const int i = (int)(t % h2);
        const int nc = (int)(t / h2);
        const int n = nc / C, c = nc - n * C;
        float v[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int s = 0; s < 4; ++s)
            if (s < nb) v[s] = ldf(y + (((size_t)n * nb + s) * C + c) * h2 * w2 + (size_t)i * w2 + j);
        T* r0 = x + ((size_t)nc * H + 2 * i) * W + 2 * j;
        stf(r0, (v[0] + v[1] + v[2] + v[3]) * 0.5f);
        stf(r0 + 1, (v[0] - v[1] + v[2] - v[3]) * 0.5f);
        stf(r0 + W, (v[0] + v[1] - v[2] - v[3]) * 0.5f);
        stf(r0 + W + 1, (v[0] - v[1] - v[2] + v[3]) * 0.5f);
    }
}

// ---------------------------------------------------------------- multi-level pyramid
// Levels 2..3 fused: a unit is a tile of 2^L rows x TW columns of one channel, loaded once;
// every level's bands are computed in registers from the level above's LL and written as
// row segments of TW / 2^l elements (naturally aligned vectors, since W % TW == 0). The
// inverse reads the deepest LL and every level's detail bands and writes the tile once.
struct PyrPtrs {
    void* p[SSBA_HAAR_MAX_LEVELS];
};

template <typename T, int n>
__device__ __forceinline__ void load_seg(const T* p, float* out)
{
    constexpr int bytes = n * (int)sizeof(T);
    if constexpr (bytes >= 16) {
#pragma unroll
        for (int q = 0; q < bytes / 16; ++q) {
            const uint4 u = __ldg(reinterpret_cast<const uint4*>(p) + q);
            if constexpr (sizeof(T) == 4) {
                float f[4];
                Lanes<float>::unpack16(u, f);
#pragma unroll
                for (int e = 0; e < 4; ++e) out[4 * q + e] = f[e];
            } else {
                float f[8];
                Lanes<__nv_bfloat16>::unpack16(u, f);
#pragma unroll
                for (int e = 0; e < 8; ++e) out[8 * q + e] = f[e];
            }
        }
    } else {
        // one naturally aligned vector of 8, 4 or 2 bytes
        if constexpr (bytes == 8) {
            float f[n];
            Lanes<T>::unpack8(__ldg(reinterpret_cast<const uint2*>(p)), f);
#pragma unroll
            for (int e = 0; e < n; ++e) out[e] = f[e];
        } else if constexpr (bytes == 4 && sizeof(T) == 2) {
            const float2 f = Lanes<__nv_bfloat16>::lo_hi(__ldg(reinterpret_cast<const unsigned int*>(p)));
            out[0] = f.x;
            out[1] = f.y;
        } else {
            out[0] = ldf(p);  // a single element
        }
    }
}

template <typename T, int n>
__device__ __forceinline__ void store_seg(T* p, const float* v)
{
    alignas(16) T tmp[n];
#pragma unroll
    for (int e = 0; e < n; ++e) {
        if constexpr (sizeof(T) == 4)
            tmp[e] = v[e];
        else
            tmp[e] = __float2bfloat16_rn(v[e]);
    }
    constexpr int bytes = n * (int)sizeof(T);
    if constexpr (bytes >= 16) {
#pragma unroll
        for (int q = 0; q < bytes / 16; ++q) reinterpret_cast<uint4*>(p)[q] = reinterpret_cast<const uint4*>(tmp)[q];
    } else if constexpr (bytes == 8) {
        *reinterpret_cast<uint2*>(p) = *reinterpret_cast<const uint2*>(tmp);
    } else if constexpr (bytes == 4) {
        *reinterpret_cast<uint32_t*>(p) = *reinterpret_cast<const uint32_t*>(tmp);
    } else {
        *reinterpret_cast<uint16_t*>(p) = *reinterpret_cast<const uint16_t*>(tmp);
    }
}

template <typename T, int L, int TW, int NB>
__global__ void __launch_bounds__(256) ssba_haar_pyr_dwt_kernel(const T* __restrict__ x, PyrPtrs y, uint32_t units,
                                                                int C, int H, int W)
{
    constexpr int TH = 1 << L;
    const uint32_t u = blockIdx.x * blockDim.x + threadIdx.x;
    if (u >= units) return;
    const uint32_t wt = W / TW, ht = H >> L;
    const uint32_t tj = u % wt, t = u / wt, ti = t % ht, nc = t / ht, n = nc / C, c = nc - n * C;
    float cur[TH][TW];
    const T* src = x + ((size_t)nc * H + (size_t)ti * TH) * W + (size_t)tj * TW;
#pragma unroll
    for (int r = 0; r < TH; ++r) load_seg<T, TW>(src + (size_t)r * W, cur[r]);
#pragma unroll
    for (int l = 1; l <= L; ++l) {
        const int rows = TH >> l, cols = TW >> l;
        const size_t hl = (size_t)(H >> l), wl = (size_t)(W >> l);
        T* yl = static_cast<T*>(y.p[l - 1]);
        float nxt[TH][TW];
#pragma unroll
        for (int r = 0; r < rows; ++r) {
            float band[4][TW];
#pragma unroll
            for (int cc = 0; cc < cols; ++cc) {
                const float p = cur[2 * r][2 * cc], q = cur[2 * r][2 * cc + 1];
                const float v = cur[2 * r + 1][2 * cc], w = cur[2 * r + 1][2 * cc + 1];
                band[0][cc] = (p + q + v + w) * 0.5f;
                band[1][cc] = (p - q + v - w) * 0.5f;
                band[2][cc] = (p + q - v - w) * 0.5f;
                band[3][cc] = (p - q - v + w) * 0.5f;
                nxt[r][cc] = band[0][cc];
            }
            const size_t off = (size_t)(ti * rows + r) * wl + (size_t)tj * cols;
#pragma unroll
            for (int s = 0; s < 4; ++s) {
                if (s < NB) {
                    T* dst = yl + (((size_t)n * NB + s) * C + c) * hl * wl + off;
                    if (cols == TW / 2) store_seg<T, TW / 2>(dst, band[s]);
                    else if (cols == TW / 4) store_seg<T, (TW / 4 > 0 ? TW / 4 : 1)>(dst, band[s]);
                    else store_seg<T, (TW / 8 > 0 ? TW / 8 : 1)>(dst, band[s]);
                }
            }
        }
#pragma unroll
        for (int r = 0; r < rows; ++r)
#pragma unroll
            for (int cc = 0; cc < cols; ++cc) cur[r][cc] = nxt[r][cc];
    }
}

template <typename T, int L, int TW, int NB>
__global__ void __launch_bounds__(256) ssba_haar_pyr_iwt_kernel(PyrPtrs y, T* __restrict__ x, uint32_t units, int C,
                                                                int H, int W)
{
    constexpr int TH = 1 << L;
    const uint32_t u = blockIdx.x * blockDim.x + threadIdx.x;
    if (u >= units) return;
    const uint32_t wt = W / TW, ht = H >> L;
    const uint32_t tj = u % wt, t = u / wt, ti = t % ht, nc = t / ht, n = nc / C, c = nc - n * C;
    // every band segment the tile needs is loaded first, the shallowest (largest) level first,
    // so that all loads are in flight together; the deepest LL is the only LL read
    float band[L][4][TH / 2][TW / 2];
#pragma unroll
    for (int l = 1; l <= L; ++l) {
        const int rows = TH >> l, cols = TW >> l;
        const size_t hl = (size_t)(H >> l), wl = (size_t)(W >> l);
        const T* yl = static_cast<const T*>(y.p[l - 1]);
#pragma unroll
        for (int r = 0; r < rows; ++r) {
            const size_t off = (size_t)(ti * rows + r) * wl + (size_t)tj * cols;
#pragma unroll
            for (int s = 0; s < 4; ++s) {
                if (s < NB && (s > 0 || l == L)) {
                    const T* srcp = yl + (((size_t)n * NB + s) * C + c) * hl * wl + off;
                    if (cols == TW / 2) load_seg<T, TW / 2>(srcp, band[l - 1][s][r]);
                    else if (cols == TW / 4) load_seg<T, (TW / 4 > 0 ? TW / 4 : 1)>(srcp, band[l - 1][s][r]);
                    else load_seg<T, (TW / 8 > 0 ? TW / 8 : 1)>(srcp, band[l - 1][s][r]);
                } else if (s > 0) {
#pragma unroll
                    for (int cc = 0; cc < cols; ++cc) band[l - 1][s][r][cc] = 0.f;  // HH with nb = 3
                }
            }
        }
    }
    float cur[TH][TW];
#pragma unroll
    for (int l = L; l >= 1; --l) {
        const int rows = TH >> l, cols = TW >> l;
        float nxt[TH][TW];
#pragma unroll
        for (int r = 0; r < rows; ++r)
#pragma unroll
            for (int cc = 0; cc < cols; ++cc) {
                const float LL = l == L ? band[l - 1][0][r][cc] : cur[r][cc];
                const float HL = band[l - 1][1][r][cc], LH = band[l - 1][2][r][cc], HH = band[l - 1][3][r][cc];
                nxt[2 * r][2 * cc] = (LL + HL + LH + HH) * 0.5f;
                nxt[2 * r][2 * cc + 1] = (LL - HL + LH - HH) * 0.5f;
                nxt[2 * r + 1][2 * cc] = (LL + HL - LH - HH) * 0.5f;
                nxt[2 * r + 1][2 * cc + 1] = (LL - HL - LH + HH) * 0.5f;
            }
#pragma unroll
        for (int r = 0; r < 2 * rows; ++r)
#pragma unroll
            for (int cc = 0; cc < 2 * cols; ++cc) cur[r][cc] = nxt[r][cc];
    }
    T* dst = x + ((size_t)nc * H + (size_t)ti * TH) * W + (size_t)tj * TW;
#pragma unroll
    for (int r = 0; r < TH; ++r) store_seg<T, TW>(dst + (size_t)r * W, cur[r]);
}

// Forward: one unit per thread with cached loads; inverse: two units per thread with
// streaming (evict-first) loads and stores -- the fastest of the shapes measured on a
// 128 x 1024 x 1024 bf16 map.
constexpr int kDwtU = 1, kIwtU = 2;
constexpr bool kDwtStream = false, kIwtStream = true;

unsigned grid_for(long long units, int per_thread)
{
    const long long want = (units + 256LL * per_thread - 1) / (256LL * per_thread);
    const long long cap = 1LL << 24;  // beyond this the grid-stride loop takes over
    return (unsigned)(want < 1 ? 1 : (want < cap ? want : cap));
}

// The band count is a template argument: with a run-time count the compiler does not batch
// the band loads, and the inverse pyramid ran three times slower.
template <typename T, int NB>
void launch_vec_nb(bool inverse, const T* in, T* out, uint32_t units, int C, int H, int W, cudaStream_t st)
{
    if (!inverse)
        ssba_haar_dwt_kernel<T, uint32_t, kDwtU, kDwtStream, NB>
            <<<grid_for(units, kDwtU), 256, 0, st>>>(in, out, units, C, H, W);
    else
        ssba_haar_iwt_kernel<T, uint32_t, kIwtU, kIwtStream, NB>
            <<<grid_for(units, kIwtU), 256, 0, st>>>(in, out, units, C, H, W);
}

template <typename T>
void launch_vec(bool inverse, const T* in, T* out, uint32_t units, int C, int H, int W, int nb, cudaStream_t st)
{
    if (nb == 4)
        launch_vec_nb<T, 4>(inverse, in, out, units, C, H, W, st);
    else
        launch_vec_nb<T, 3>(inverse, in, out, units, C, H, W, st);
}

template <typename T>
int launch_haar_t(bool inverse, const void* in, void* out, int N, int C, int H, int W, int nb, cudaStream_t st)
{
    constexpr int V = Lanes<T>::V;
    const int NC = N * C;
    if (W % (2 * V) == 0) {
        // 32-bit unit indices: launch whole images in groups of fewer than 2^31 units
        const long long per_image = (long long)C * (H / 2) * (W / (2 * V));
        if (per_image >= (1LL << 31)) {
            set_error("ssba_haar: one image of %lld vector units exceeds the 2^31 limit", per_image);
            return SSBA_ERR_UNSUPPORTED;
        }
        const int group = (int)std::min<long long>(N, ((1LL << 31) - 1) / per_image);
        const size_t x_image = (size_t)C * H * W;              // elements of one image
        const size_t y_image = (size_t)nb * C * (H / 2) * (W / 2);  // elements of its bands
        for (int n0 = 0; n0 < N; n0 += group) {
            const int g = std::min(group, N - n0);
            const T* src = static_cast<const T*>(in) + (size_t)n0 * (inverse ? y_image : x_image);
            T* dst = static_cast<T*>(out) + (size_t)n0 * (inverse ? x_image : y_image);
            launch_vec<T>(inverse, src, dst, (uint32_t)(g * per_image), C, H, W, nb, st);
        }
    } else {
        const long long units = (long long)NC * (H / 2) * (W / 2);
        const unsigned grid = grid_for(units, 1);
        if (!inverse)
            ssba_haar_dwt_scalar_kernel<T><<<grid, 256, 0, st>>>(static_cast<const T*>(in), static_cast<T*>(out), NC, C,
                                                                H, W, nb);
        else
            ssba_haar_iwt_scalar_kernel<T><<<grid, 256, 0, st>>>(static_cast<const T*>(in), static_cast<T*>(out), NC, C,
                                                                H, W, nb);
    }
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) {
        set_error("ssba_haar launch: %s", cudaGetErrorString(e));
        return SSBA_ERR_CUDA;
    }
    return SSBA_OK;
}

template <typename T, int L, int TW, int NB>
void launch_pyr_nb(bool inverse, const T* x, T* xo, const PyrPtrs& y, uint32_t units, int C, int H, int W,
                   cudaStream_t st)
{
    const unsigned grid = (units + 255) / 256;
    if (!inverse)
        ssba_haar_pyr_dwt_kernel<T, L, TW, NB><<<grid, 256, 0, st>>>(x, y, units, C, H, W);
    else
        ssba_haar_pyr_iwt_kernel<T, L, TW, NB><<<grid, 256, 0, st>>>(y, xo, units, C, H, W);
}

template <typename T, int L, int TW>
void launch_pyr_tw(bool inverse, const T* x, T* xo, const PyrPtrs& y, uint32_t units, int C, int H, int W, int nb,
                   cudaStream_t st)
{
    if (nb == 4)
        launch_pyr_nb<T, L, TW, 4>(inverse, x, xo, y, units, C, H, W, st);
    else
        launch_pyr_nb<T, L, TW, 3>(inverse, x, xo, y, units, C, H, W, st);
}

template <typename T>
int launch_pyr_t(bool inverse, void* x, void* const* ys, int N, int C, int H, int W, int L, int nb, cudaStream_t st)
{
    // widest tile: 16 bytes of a row, and at least 2^L columns; else 2^L columns
    const int tw_vec = std::max(1 << L, 16 / (int)sizeof(T));
    const int TW = (W % tw_vec == 0) ? tw_vec : (1 << L);
    const long long per_image = (long long)C * (H >> L) * (W / TW);
    if (per_image >= (1LL << 31)) {
        set_error("ssba_haar pyramid: one image of %lld tiles exceeds the 2^31 limit", per_image);
        return SSBA_ERR_UNSUPPORTED;
    }
    const int group = (int)std::min<long long>(N, ((1LL << 31) - 1) / per_image);
    const size_t x_image = (size_t)C * H * W;
    for (int n0 = 0; n0 < N; n0 += group) {
        const int g = std::min(group, N - n0);
        T* xp = static_cast<T*>(x) + (size_t)n0 * x_image;
        PyrPtrs y{};
        for (int l = 1; l <= L; ++l)
            y.p[l - 1] = static_cast<T*>(ys[l - 1]) + (size_t)n0 * nb * C * (size_t)(H >> l) * (size_t)(W >> l);
        const uint32_t units = (uint32_t)(g * per_image);
        if (L == 2 && TW == 4) launch_pyr_tw<T, 2, 4>(inverse, xp, xp, y, units, C, H, W, nb, st);
        else if (L == 2 && TW == 8) launch_pyr_tw<T, 2, 8>(inverse, xp, xp, y, units, C, H, W, nb, st);
        else if (L == 3 && TW == 8) launch_pyr_tw<T, 3, 8>(inverse, xp, xp, y, units, C, H, W, nb, st);
        else {
            set_error("ssba_haar pyramid: no kernel for %d levels with %d-column tiles", L, TW);
            return SSBA_ERR_UNSUPPORTED;
        }
    }
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) {
        set_error("ssba_haar pyramid launch: %s", cudaGetErrorString(e));
        return SSBA_ERR_CUDA;
    }
    return SSBA_OK;
}

}  // namespace

int launch_haar(bool inverse, const void* in, void* out, int N, int C, int H, int W, int nb, int dtype,
                cudaStream_t st)
{
    return dtype == SSBA_BF16 ? launch_haar_t<__nv_bfloat16>(inverse, in, out, N, C, H, W, nb, st)
                              : launch_haar_t<float>(inverse, in, out, N, C, H, W, nb, st);
}

}  // namespace ssba

namespace ssba {

int launch_haar_pyramid(bool inverse, void* x, void* const* ys, int N, int C, int H, int W, int L, int nb, int dtype,
                        cudaStream_t st)
{
    if (L == 1)
        return inverse ? launch_haar(true, ys[0], x, N, C, H, W, nb, dtype, st)
                       : launch_haar(false, x, ys[0], N, C, H, W, nb, dtype, st);
    return dtype == SSBA_BF16 ? launch_pyr_t<__nv_bfloat16>(inverse, x, ys, N, C, H, W, L, nb, st)
                              : launch_pyr_t<float>(inverse, x, ys, N, C, H, W, L, nb, st);
}

}  // namespace ssba
