// Host-side helpers shared by the library's translation units.
#pragma once
#include <cstdarg>
#include <cstdint>
#include <cstdio>

#include "../../include/jnx.h"

namespace jnx {

// Record a printf-style message for jnx_last_error() and return `code`.
jnx_status fail(jnx_status code, const char* fmt, ...);
void clear_error();

}  // namespace jnx
