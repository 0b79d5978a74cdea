// tcgen05 (5th-generation tensor core) kernels: placeholder translation unit.
#include "pnn_internal.h"
