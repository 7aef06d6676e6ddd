/*
 * Oracle (test infrastructure only): IEEE binary16 rounding, from the format's
 * definition. The method stores its row/column scales and its pivot values in
 * FP16 (App. C.3 step 6, App. D).
 */
#include <math.h>
#include "oracle.h"

/* Round x to the nearest binary16 value, ties to even. Values beyond the
 * largest finite binary16 (65504) saturate to +-65504 instead of overflowing:
 * the stored state stays finite. Subnormal binary16 values (below 2^-14) are
 * produced with their fixed quantum 2^-24. NaN passes through. */
double or_fp16_round(double x)
{
    if (x == 0.0 || isnan(x))
        return x;
    double a = fabs(x);
    if (a >= 65504.0)
        return copysign(65504.0, x);
    int e;
    frexp(a, &e);                /* a in [2^(e-1), 2^e) */
    int E = e - 1;
    if (E < -14)
        E = -14;                 /* subnormal range shares the quantum of 2^-14 */
    double quantum = ldexp(1.0, E - 10);  /* 10 fraction bits */
    double n = nearbyint(a / quantum);    /* exact quotient; default mode is ties-to-even */
    double r = n * quantum;
    if (r > 65504.0)
        r = 65504.0;
    return copysign(r, x);
}

/* Bit pattern of a value that is exactly representable in binary16. */
uint16_t or_fp16_encode(double v)
{
    if (isnan(v))
        return 0x7E00;
    uint16_t s = signbit(v) ? 0x8000 : 0;
    double a = fabs(v);
    if (a == 0.0)
        return s;
    if (isinf(v))
        return s | 0x7C00;
    if (a < ldexp(1.0, -14))
        return s | (uint16_t)(a / ldexp(1.0, -24));   /* subnormal: fraction counts 2^-24 */
    int e;
    double m = frexp(a, &e);                           /* a = m 2^e, m in [0.5, 1) */
    int E = e - 1;
    uint16_t frac = (uint16_t)((2.0 * m - 1.0) * 1024.0);
    return s | (uint16_t)((E + 15) << 10) | frac;
}

double or_fp16_decode(uint16_t h)
{
    int s = h >> 15, E = (h >> 10) & 0x1F, f = h & 0x3FF;
    double v;
    if (E == 0)
        v = ldexp((double)f, -24);
    else if (E == 31)
        v = f ? NAN : INFINITY;
    else
        v = ldexp(1.0 + f / 1024.0, E - 15);
    return s ? -v : v;
}
