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
template <typename T, typename I, int U, bool kStream>
__global__ void __launch_bounds__(256) ssba_haar_dwt_kernel(const T* __restrict__ x, T* __restrict__ y, I units,
                                                            int C, int H, int W, int nb)
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
                dst[k] = ((size_t)n * nb * C + c) * h2 * w2 + (size_t)i * w2 + V * jv;
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
                    if (s < nb) st<kStream>(reinterpret_cast<uint2*>(y + dst[k] + s * plane), Lanes<T>::pack8(band[s]));
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
template <typename T, typename I, int U, bool kStream>
__global__ void __launch_bounds__(256) ssba_haar_iwt_kernel(const T* __restrict__ y, T* __restrict__ x, I units,
                                                            int C, int H, int W, int nb)
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
                const T* src = y + ((size_t)n * nb * C + c) * h2 * w2 + (size_t)i * w2 + V * jv;
#pragma unroll
                for (int s = 0; s < 4; ++s)
                    rv[k][s] = s < nb ? ld<kStream>(reinterpret_cast<const uint2*>(src + s * plane)) : make_uint2(0u, 0u);
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

template <typename T>
void launch_vec(bool inverse, const T* in, T* out, uint32_t units, int C, int H, int W, int nb, cudaStream_t st)
{
    if (!inverse)
        ssba_haar_dwt_kernel<T, uint32_t, kDwtU, kDwtStream>
            <<<grid_for(units, kDwtU), 256, 0, st>>>(in, out, units, C, H, W, nb);
    else
        ssba_haar_iwt_kernel<T, uint32_t, kIwtU, kIwtStream>
            <<<grid_for(units, kIwtU), 256, 0, st>>>(in, out, units, C, H, W, nb);
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

}  // namespace

int launch_haar(bool inverse, const void* in, void* out, int N, int C, int H, int W, int nb, int dtype,
                cudaStream_t st)
{
    return dtype == SSBA_BF16 ? launch_haar_t<__nv_bfloat16>(inverse, in, out, N, C, H, W, nb, st)
                              : launch_haar_t<float>(inverse, in, out, N, C, H, W, nb, st);
}

}  // namespace ssba
